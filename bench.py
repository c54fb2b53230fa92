#!/usr/bin/env python3
"""Benchmark of the STaR-KV compression step on GB300.

One step = Algorithm 1 for every layer of the workload: window-query scoring
(two tcgen05 passes), online MI / temporal / entropy calibration, global top-B
and the KV gather, through the C ABI (``starkv_step``).  Default workload: 28
layers of the 5-screenshot UI-TARS-1.5-7B shape (28 q heads / 4 KV heads,
d = 128, w = 32, 5 x 2704 visual + 512 text tokens, B = 20% of visual).

Prints ONE JSON line (rank 0).  ``value`` is cache tokens scored per second
(sum over layers and sequences of L_past per step / step time), inputs resident
in HBM; ``e2e`` is the same metric through ``starkv_step_host`` with pinned
host buffers, copies inside the timed region.  ``--impl reference`` times the
fp64 CPU oracle on the same workload instead.

Multi-GPU (torchrun): each rank compresses its own independent trajectory
(weak scaling, no collective on the data path); timing is max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time
from pathlib import Path

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

METRIC = "KV compression latency/step (ms) & cache tokens scored/s; % of HBM/TC roofline"
UNIT = "tokens/s"


def _peaks():
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        d = json.loads(p.read_text())
        return dict(hbm=float(d["hbm_gbs"]), tc=float(d["bf16_tflops"]),
                    tc_sus=float(d.get("bf16_tflops_sustained", d["bf16_tflops"])), src="measured")
    return dict(hbm=6800.0, tc=1900.0, tc_sus=1700.0, src="fallback")


# ----------------------------------------------------------------------------- work accounting

def work_per_step(wl, seqs, per_head=False):
    """Algorithmic bytes and flops of one step, per kernel kind and in total.

    Per scored token and layer: K read once (G * d * 2 B) and 2 * H * w * d
    flop of Q K^T; per (layer, seq): window queries H * w * d * 2 B; the group
    score map written and read (2 * G * 4 B per token); per kept row: K and V
    read and written (4 * G * d * 2 B) and its metadata word read and written
    (once, or once per group in the per-KV-head mode)."""
    H, G, w, d, nl = wl.n_heads, wl.n_kv_heads, wl.window, wl.head_dim, wl.n_layers
    tok = sum(s["L"] - w for s in seqs) * nl
    kept = sum(s["B"] + w for s in seqs) * nl
    qk_flops = 2.0 * H * w * d * tok
    k_bytes = G * d * 2.0 * tok + H * w * d * 2.0 * nl * len(seqs)
    s_bytes = 2 * G * 4.0 * tok
    gather = 4.0 * G * d * 2 * kept + 2 * 4.0 * kept * (G if per_head else 1)
    return dict(tokens=tok, qk_flops=qk_flops, k_bytes=k_bytes, s_bytes=s_bytes, gather_bytes=gather,
                step_bytes=k_bytes + s_bytes + gather)


def with_attention(wl, work, n_seqs):
    """The step's work when it also runs the window-attention producer (the
    model's own attention of the window rows, whose normaliser the compression
    then takes): V read once (G * d * 2 B per scored token and layer) and the
    output written (H * w * d fp32 per layer and sequence) on top of K and Q,
    and the P V flops (as many as Q K^T) on top of Q K^T."""
    v_bytes = wl.n_kv_heads * wl.head_dim * 2.0 * work["tokens"]
    o_bytes = wl.n_heads * wl.window * wl.head_dim * 4.0 * wl.n_layers * n_seqs
    out = dict(work)
    out["attn_bytes"] = work["k_bytes"] + v_bytes + o_bytes
    out["step_bytes"] = work["step_bytes"] + v_bytes + o_bytes
    out["step_flops"] = 2 * work["qk_flops"]
    return out


def kernel_work(kind, work, peaks):
    """(bound, algorithmic units per step, unit) of one kernel kind.  A scoring
    pass reads K once and does the Q K^T flops; its bound is whichever of the
    two takes longer at the measured peaks (224 flop per byte at the UI-TARS
    shape, below the HBM / bf16 ridge, so HBM)."""
    if kind in ("score_lse", "score_accum"):
        t_hbm = work["k_bytes"] / (peaks["hbm"] * 1e9)
        t_tc = work["qk_flops"] / (peaks["tc_sus"] * 1e12)
        if t_hbm >= t_tc:
            return "hbm", work["k_bytes"] / 1e9, "GB/s"
        return "tensor", work["qk_flops"] / 1e12, "TFLOP/s"
    if kind == "compact":
        return "hbm", work["gather_bytes"] / 1e9, "GB/s"
    if kind == "attention":
        return "hbm", work["attn_bytes"] / 1e9, "GB/s"
    return "hbm", work["s_bytes"] / 1e9, "GB/s"


def code_only(text):
    """C/C++ source without its comments and with whitespace runs collapsed,
    so that an edit of comments alone keeps a kernel's recorded counters."""
    out, i, n = [], 0, len(text)
    while i < n:
        c = text[i]
        if c in "\"'":   # string or character literal, copied as is
            j = i + 1
            while j < n and text[j] != c:
                j += 2 if text[j] == "\\" else 1
            out.append(text[i:j + 1])
            i = j + 1
        elif text.startswith("//", i):
            j = text.find("\n", i)
            i = n if j < 0 else j
        elif text.startswith("/*", i):
            j = text.find("*/", i + 2)
            i = n if j < 0 else j + 2
            out.append(" ")
        else:
            out.append(c)
            i += 1
    return " ".join("".join(out).split())


def kernel_src_hash(kind, read=None):
    """Hash of the code (comments excluded) that a kernel is built from;
    ``read(name)`` returns a source file's text (default: the working tree)."""
    files = {"score_lse": "score.cu", "score_accum": "score.cu", "pool": "score.cu",
             "calibrate": "select.cu", "compact": "compact.cu", "attention": "attn.cu",
             "attn_combine": "attn.cu"}[kind]
    read = read or (lambda f: (ROOT / "paper_2606_01790_gb300" / "csrc" / f).read_text())
    h = hashlib.sha256()
    for f in (files, "ptx.cuh", "common.cuh"):
        h.update(code_only(read(f)).encode())
    return h.hexdigest()[:16]


def recorded_traffic(kind, workload):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current source of the kernel; else None."""
    p = ROOT / "profiles" / "traffic.json"
    if not p.exists():
        return None
    d = json.loads(p.read_text()).get(f"{kind}@{workload}")
    if not d or d.get("src_sha") != kernel_src_hash(kind):
        return None
    return d.get("dram_bytes_per_launch")


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.samples = []
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(device_index)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        self.t = threading.Thread(target=self._read, daemon=True)
        self.t.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), [x.strip() for x in line.split(",")]))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0, t1):
        rows = [s for (t, s) in self.samples if t0 <= t <= t1]
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4)
                          if len(r) > 5 + i and r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows),
                "power_w_max": max((num(r[3]) or 0.0) for r in rows)}


# ----------------------------------------------------------------------------- oracle (CPU)

def oracle_worker(args):
    """Times the fp64 oracle on the workload; prints one JSON line.

    Layers 0, 1, ... of sequence 0 (step 0 of the workload), cycled: either
    ``--repeat`` layer compressions (the reference arm's steps) or, with
    ``--repeat 0``, until ``--budget-s`` seconds of oracle work have run.
    ``--budget-pct`` overrides the workload's budget as in the GPU arm."""
    from oracle import starkv_oracle as O
    from paper_2606_01790_gb300 import synthetic as syn
    wl = syn.WORKLOADS[args.workload]
    p = O.Params()
    per_head = args.select_mode == "per_head"
    spent, tokens = 0.0, 0
    per_call, layers_done = [], []
    nl = min(wl.n_layers, args.max_layers)
    layers = (i % nl for i in range(args.repeat if args.repeat > 0 else 1 << 30))
    cache = {}
    for layer in layers:
        if layer not in cache:
            si = syn.make_sequence(wl, seq=0, layers=[layer])
            if args.budget_pct:
                si.budget = syn.budget(args.budget_pct, si.n_visual_history, si.L - wl.window)
            cache = {layer: si}   # one layer's inputs held at a time
        si = cache[layer]
        lay = si.layout[0]
        st = O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols)
        q, k, v = si.q[0].double().numpy(), si.k[0].double().numpy(), si.v[0].double().numpy()
        t = time.perf_counter()
        O.step_layer(q, k, v, lay.is_visual, lay.frame, lay.row, lay.col, si.cur_frame, si.budget,
                     wl.window, wl.grid_rows, wl.grid_cols, st, p, per_head=per_head)
        dt = time.perf_counter() - t
        per_call.append(dt)
        layers_done.append(layer)
        spent += dt
        tokens += si.L - wl.window
        if args.repeat == 0 and spent >= args.budget_s:
            break
    print(json.dumps(dict(tokens=tokens, seconds=spent, calls=len(per_call), per_call=per_call,
                          layers=layers_done, l_past=si.L - wl.window, n_layers=wl.n_layers)))


def run_oracle_subprocess(workload, budget_s=15.0, max_layers=28, repeat=0, select_mode="global",
                          threads=None, budget_pct=0):
    """The oracle worker in a child process with ``threads`` BLAS threads
    (default: all host cores)."""
    threads = str(threads or os.cpu_count() or 1)
    env = dict(os.environ, OPENBLAS_NUM_THREADS=threads, OMP_NUM_THREADS=threads,
               MKL_NUM_THREADS=threads, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, str(ROOT / "bench.py"), "--oracle-worker", "--workload", workload,
                        "--budget-s", str(budget_s), "--max-layers", str(max_layers),
                        "--repeat", str(repeat), "--select-mode", select_mode,
                        "--budget-pct", str(budget_pct)],
                       capture_output=True, text=True, env=env, timeout=3600)
    if r.returncode != 0:
        raise RuntimeError(f"oracle worker failed:\n{r.stderr[-2000:]}")
    d = json.loads(r.stdout.strip().splitlines()[-1])
    d["cores"] = int(threads)
    return d


def seconds_text(t):
    """A duration in s, or in ms below one second."""
    return f"{t:.1f} s" if t >= 1.0 else f"{1e3 * t:.1f} ms"


def oracle_sample(d, what):
    """Words for a timed oracle sample, with the whole-step extrapolation."""
    per_layer = d["seconds"] / max(1, d["calls"])
    return (f"{what}: {d['calls']} layer compressions of sequence 0 (layers "
            f"{min(d['layers'])}..{max(d['layers'])} cycled, step 0 of the workload), {d['tokens']} "
            f"tokens scored in {d['seconds']:.1f} s, numpy BLAS on {d['cores']} thread(s); a whole "
            f"{d['n_layers']}-layer step extrapolates to {seconds_text(d['n_layers'] * per_layer)} at this rate")


def cpu_baselines(args):
    """The oracle timed on the host cores: all cores (the reported
    cpu_baseline) and one thread, each on a bounded sample."""
    sel = args.select_mode
    o = run_oracle_subprocess(args.workload, budget_s=args.cpu_budget_s, select_mode=sel,
                              budget_pct=args.budget_pct)
    one = run_oracle_subprocess(args.workload, budget_s=args.cpu_budget_s / 2, select_mode=sel, threads=1,
                                budget_pct=args.budget_pct)
    cpu = {"value": o["tokens"] / o["seconds"], "unit": UNIT, "cores": o["cores"], "kind": "oracle",
           "sample": oracle_sample(o, "all host cores")}
    cpu1 = {"value": one["tokens"] / one["seconds"], "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": oracle_sample(one, "one thread")}
    return cpu, cpu1


def reference_arm(args):
    """--impl reference: the fp64 oracle as it stands, one layer of the
    workload per step (layer = step mod n_layers), on the host cores (rank 0
    only)."""
    if rank_env()[1] != 0:
        return
    from paper_2606_01790_gb300 import synthetic as syn
    wl = syn.WORKLOADS[args.workload]
    d = run_oracle_subprocess(args.workload, repeat=args.warmup + args.steps, select_mode=args.select_mode,
                              budget_pct=args.budget_pct)
    times = d["per_call"][args.warmup:]
    toks = d["tokens"] * len(times) / max(1, d["calls"])   # the same L_past in every layer
    total = sum(times)
    value = toks / total
    sample = (f"one layer compression per step (layer = step mod {wl.n_layers}, sequence 0, step 0 of the "
              f"workload; L_past = {d['l_past']} tokens scored per step), numpy BLAS on {d['cores']} "
              f"threads; a whole {wl.n_layers}-layer step extrapolates to "
              f"{seconds_text(wl.n_layers * total / len(times))} at this rate")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * total / len(times), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": args.workload, "select_mode": args.select_mode,
                   "budget_pct": args.budget_pct or None},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": d["cores"], "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


# ----------------------------------------------------------------------------- ranks

def rank_env():
    """(world size, rank, local rank) from the torchrun environment."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def rank_seeds(rank, n_seqs):
    """Each rank compresses its own trajectories (weak scaling): distinct seeds."""
    return [rank * 1000 + i for i in range(n_seqs)]


def max_over_ranks(x, dist, device):
    """The largest value of ``x`` over all ranks (the job's time is its slowest rank's)."""
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    if dist is not None:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_rank_step, world, steps, ms_max):
    """Whole-job tokens/s: every rank's tokens over the slowest rank's time."""
    return tokens_per_rank_step * world * steps / (ms_max / 1e3)


# ----------------------------------------------------------------------------- GPU arm

class GpuBench:
    """Device set-up, inputs and the timed loops of the GPU arm."""

    def __init__(self, args):
        import torch
        import __graft_entry__
        from paper_2606_01790_gb300 import starkv as sk
        from paper_2606_01790_gb300 import synthetic as syn
        self.torch, self.sk, self.syn, self.args = torch, sk, syn, args
        self.world, self.rank, local = rank_env()
        self.dist = None
        if self.world > 1:
            import torch.distributed as dist
            dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
            self.dist = dist
        torch.cuda.set_device(local)
        self.local = local
        self.dev = torch.device("cuda", local)
        __graft_entry__.build()
        self.wl = syn.WORKLOADS[args.workload]
        self.peaks = _peaks()
        self.step_fn = sk.step

    def use_attention(self):
        """Every step first runs the window-attention producer, whose
        normalisers the compression step then takes (its first scoring pass
        skipped): the model's attention of the window rows plus the
        compression, as App. A.3 accounts them."""
        sk = self.sk

        def step(st, seqs, ws):
            sk.window_attention(st, seqs, ws)
            sk.step(st, seqs, ws)
        self.step_fn = step

    def config(self, n_seqs):
        sk, wl = self.sk, self.wl
        return sk.Config(n_layers=wl.n_layers, n_heads=wl.n_heads, n_kv_heads=wl.n_kv_heads,
                         head_dim=wl.head_dim, window=wl.window, grid_rows=wl.grid_rows,
                         grid_cols=wl.grid_cols, max_seqs=n_seqs,
                         select_mode=sk.SELECT_PER_HEAD if self.args.select_mode == "per_head"
                         else sk.SELECT_GLOBAL)

    def with_budget(self, si):
        if self.args.budget_pct:
            si.budget = self.syn.budget(self.args.budget_pct, si.n_visual_history, si.L - self.wl.window)
        return si

    def make_seq(self, si, slot, P, pin=False):
        """Device (or page-locked host) buffers of one sequence."""
        torch, sk, wl = self.torch, self.sk, self.wl
        G, w, d, nl = wl.n_kv_heads, wl.window, wl.head_dim, wl.n_layers
        L, B = si.L, si.budget
        words = sk.pack_meta(si.layout[0].is_visual, si.layout[0].frame, si.layout[0].row, si.layout[0].col)
        alloc = (lambda shape, dt: torch.empty(shape, dtype=dt, pin_memory=True)) if pin else \
            (lambda shape, dt: torch.empty(shape, dtype=dt, device=self.dev))

        def put(t):
            if pin:
                o = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
                o.copy_(t)
                return o
            return t.to(self.dev)
        return sk.Seq(k=put(si.k), v=put(si.v), q=put(si.q), meta=put(sk.meta_tensor(words)),
                      meta_layer_stride=0, L=L, cur_frame=si.cur_frame, budget=B, slot=slot,
                      k_out=alloc((nl, G, B + w, d), torch.bfloat16),
                      v_out=alloc((nl, G, B + w, d), torch.bfloat16),
                      meta_out=alloc((nl, P, B + w), torch.int32), idx=alloc((nl, P, B), torch.int32))

    def barrier(self):
        if self.dist is not None:
            self.dist.barrier()
        self.torch.cuda.synchronize(self.dev)

    def time_steps(self, st, seqs, ws, steps, warmup, soak_s=0.0):
        """Device ms of ``steps`` back-to-back starkv_step calls (CUDA events on
        the launch stream), after ``warmup`` untimed steps and a soak; the
        launches made in the timed region."""
        torch, sk = self.torch, self.sk
        for _ in range(warmup):
            self.step_fn(st, seqs, ws)
        torch.cuda.synchronize(self.dev)
        sk.check_device_error(st)
        t_soak = time.time()
        while time.time() - t_soak < soak_s:
            for _ in range(10):
                self.step_fn(st, seqs, ws)
            torch.cuda.synchronize(self.dev)
        sk.kernel_times(st)   # reset counters
        self.barrier()
        stream = torch.cuda.current_stream(self.dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            self.step_fn(st, seqs, ws)
        e1.record(stream)
        self.barrier()
        ms = e0.elapsed_time(e1)
        launches = sum(v[0] for v in sk.kernel_times(st).values())   # kept with timing off
        sk.check_device_error(st)
        return ms, launches

    def kernel_pass(self, st, seqs, ws, n):
        """Per-kernel device times in a separate pass: the event pair around
        every launch keeps the next kernel from starting under the previous
        one's tail.  {kind: (launches, total_ms)}."""
        torch, sk = self.torch, self.sk
        sk.set_timing(st, True)
        for _ in range(n):
            self.step_fn(st, seqs, ws)
        torch.cuda.synchronize(self.dev)
        sk.set_timing(st, False)
        return sk.kernel_times(st)

    def e2e(self, st, sis, P, n, devseqs):
        """The same metric through starkv_step_host (page-locked host buffers,
        copies in the timed region): (ms per step, h2d bytes, d2h bytes)."""
        torch, sk = self.torch, self.sk
        hseqs = [self.make_seq(si, i, P, pin=True) for i, si in enumerate(sis)]
        for hs_, s_ in zip(hseqs, devseqs):
            if s_.lse is not None:
                hs_.lse = torch.empty(s_.lse.shape, dtype=torch.float32, pin_memory=True)
                hs_.lse.copy_(s_.lse)
        hws = sk.workspace(st, hseqs, host=True, device=self.dev)
        # K, Q and metadata are uploaded; V is page-locked, so the gather reads
        # only its kept rows in place (the same bytes as V')
        h2d = sum(s.k.numel() * 2 + s.v_out.numel() * 2 + s.q.numel() * 2 + s.meta.numel() * 4 +
                  (s.lse.numel() * 4 if s.lse is not None else 0) for s in hseqs)
        d2h = sum(s.k_out.numel() * 2 + s.v_out.numel() * 2 + s.meta_out.numel() * 4 + s.idx.numel() * 4
                  for s in hseqs)
        for _ in range(2):
            sk.step_host(st, hseqs, hws)
        self.barrier()
        stream = torch.cuda.current_stream(self.dev)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n):
            sk.step_host(st, hseqs, hws)
        b.record(stream)
        self.barrier()
        e_ms = max_over_ranks(a.elapsed_time(b), self.dist, self.dev)
        sk.check_device_error(st)
        return e_ms / n, h2d, d2h

    def e2e_attention(self, st, sis, P, n, devseqs, ws):
        """The end-to-end step with the attention producer: K, V, Q and the
        metadata copied from page-locked host buffers, the producer and the
        step on the device buffers, the compacted cache and indices copied
        back, all in the timed region: (ms per step, h2d bytes, d2h bytes)."""
        torch, sk = self.torch, self.sk
        hseqs = [self.make_seq(si, i, P, pin=True) for i, si in enumerate(sis)]
        names_in, names_out = ("k", "v", "q", "meta"), ("k_out", "v_out", "meta_out", "idx")
        h2d = sum(getattr(h, a).numel() * getattr(h, a).element_size() for h in hseqs for a in names_in)
        d2h = sum(getattr(h, a).numel() * getattr(h, a).element_size() for h in hseqs for a in names_out)

        def one():
            for h, d in zip(hseqs, devseqs):
                for a in names_in:
                    getattr(d, a).copy_(getattr(h, a), non_blocking=True)
            sk.window_attention(st, devseqs, ws)
            sk.step(st, devseqs, ws)
            for h, d in zip(hseqs, devseqs):
                for a in names_out:
                    getattr(h, a).copy_(getattr(d, a), non_blocking=True)
        for _ in range(2):
            one()
        self.barrier()
        stream = torch.cuda.current_stream(self.dev)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n):
            one()
        b.record(stream)
        self.barrier()
        e_ms = max_over_ranks(a.elapsed_time(b), self.dist, self.dev)
        sk.check_device_error(st)
        return e_ms / n, h2d, d2h

    def roofline(self, kt, work, n_kt, workload):
        """The dominant kernel's achieved rate against its binding peak, and its
        share of the per-kernel pass."""
        kernels = {}
        total = max(1e-9, sum(v[1] for v in kt.values()))
        for kind, (n, tms) in kt.items():
            if n:
                kernels[kind] = {"launches": n, "avg_us": 1e3 * tms / n, "share": tms / total}
        dom = max(kernels, key=lambda k: kernels[k]["avg_us"] * kernels[k]["launches"])
        bound, units_per_step, unit = kernel_work(dom, work, self.peaks)
        per_launch = units_per_step * n_kt / kernels[dom]["launches"]
        achieved = per_launch / (kernels[dom]["avg_us"] * 1e-6)
        peak = self.peaks["tc_sus"] if bound == "tensor" else self.peaks["hbm"]
        roof = {"bound": bound, "achieved": achieved, "peak": peak, "unit": unit, "frac": achieved / peak,
                "traffic": recorded_traffic(dom, workload), "kernel": dom,
                "scope": "the dominant kernel alone; the whole step's fraction is step_roofline.frac",
                "peak_src": f"{self.peaks['src']} ({'bf16 sustained' if bound == 'tensor' else 'HBM copy'})"}
        return roof, kernels

    def step_roofline(self, work, ms_step):
        flops = work.get("step_flops", work["qk_flops"])
        us = max(work["step_bytes"] / (self.peaks["hbm"] * 1e9), flops / (self.peaks["tc"] * 1e12)) * 1e6
        return {"roofline_us": us, "measured_us": 1e3 * ms_step, "frac": us / (1e3 * ms_step),
                "alg_bytes": work["step_bytes"], "alg_flops": flops, "peak_src": self.peaks["src"]}


def gpu_arm(args):
    gb = GpuBench(args)
    if args.trajectory:
        return trajectory_arm(gb)
    torch, sk, syn, wl = gb.torch, gb.sk, gb.syn, gb.wl
    seeds = rank_seeds(gb.rank, wl.n_seqs)
    sis = [gb.with_budget(syn.make_sequence(wl, seq=i, seed=s)) for i, s in enumerate(seeds)]
    st = sk.init_state(gb.config(len(sis)))
    P = sk.sel_rows(st.cfg)   # rows of idx / meta_out per layer
    seqs = [gb.make_seq(si, i, P) for i, si in enumerate(sis)]
    work = work_per_step(wl, [dict(L=si.L, B=si.budget) for si in sis], per_head=P > 1)
    if args.lse == "given":
        # every step runs the window-attention producer (the model's own
        # attention of the window rows, output and normalisers), and the
        # compression takes its normalisers
        for s_ in seqs:
            s_.attn_o = torch.empty((wl.n_layers, wl.n_heads, wl.window, wl.head_dim), dtype=torch.float32,
                                    device=gb.dev)
            s_.attn_lse = torch.empty((wl.n_layers, wl.n_heads, wl.window), dtype=torch.float32, device=gb.dev)
            s_.lse = s_.attn_lse
        gb.use_attention()
        work = with_attention(wl, work, len(seqs))
    ws = sk.workspace(st, seqs, device=gb.dev)

    clocks = ClockSampler(gb.local)
    t0 = time.time()
    ms, launches = gb.time_steps(st, seqs, ws, args.steps, args.warmup, args.soak_s)
    t_end = time.time()
    clocks.stop()
    ms_max = max_over_ranks(ms, gb.dist, gb.dev)
    ms_step = ms_max / args.steps
    value = job_throughput(work["tokens"], gb.world, args.steps, ms_max)
    n_kt = max(1, min(args.steps, 20))
    roofline, kernels = gb.roofline(gb.kernel_pass(st, seqs, ws, n_kt), work, n_kt, args.workload)
    step_roofline = gb.step_roofline(work, ms_step)

    e2e = None
    if not args.no_e2e:
        n_e2e = max(1, min(args.steps, 20))
        if args.lse == "given":
            e_ms, h2d, d2h = gb.e2e_attention(st, sis, P, n_e2e, seqs, ws)
        else:
            e_ms, h2d, d2h = gb.e2e(st, sis, P, n_e2e, seqs)
        e2e = {"value": job_throughput(work["tokens"], gb.world, 1, e_ms), "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": n_e2e, "ms_per_step": e_ms}

    cpu = cpu1 = None
    if gb.rank == 0 and gb.world == 1 and not args.no_cpu_baseline:
        cpu, cpu1 = cpu_baselines(args)

    if gb.rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": gb.world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": args.workload, "select_mode": args.select_mode,
                       "lse": "from the window-attention producer run in every step (the model's attention "
                              "of the window rows: output and normalisers); first scoring pass skipped"
                       if args.lse == "given" else "computed (both scoring passes)", "layers": wl.n_layers, "seqs_per_gpu": len(sis),
                       "L": [si.L for si in sis], "w": wl.window, "B": [si.budget for si in sis],
                       "budget_pct": args.budget_pct or None, "H": wl.n_heads, "G": wl.n_kv_heads,
                       "d": wl.head_dim,
                       "l2": f"inputs {2 * sum(s.k.numel() for s in seqs) * 2 / 1e9:.2f} GB per step "
                             "> 129 MB L2 (no flush)",
                       "parallelism": f"replicas x{gb.world}"},
            "step_roofline": step_roofline, "roofline": roofline, "kernels": kernels,
            "cpu_baseline": cpu, "cpu_baseline_1thread": cpu1, "e2e": e2e, "gpu_launches": launches,
            "clocks": clocks.summary(t0, t_end),
        }))
    if gb.dist is not None:
        gb.dist.destroy_process_group()
    st.close()


def trajectory_arm(gb):
    """Config 3 as a trajectory: step s compresses the cache that step s - 1's
    own compaction produced plus one new screenshot and its text, with the
    temporal and MI state carried.  Each step is timed on its own input: the
    slot's state is saved before the timed repeats and restored after them,
    then the step runs once more to produce the next step's cache."""
    import numpy as np
    args, torch, sk, syn, wl = gb.args, gb.torch, gb.sk, gb.syn, gb.wl
    if wl.steps <= 1 or args.select_mode != "global":
        raise SystemExit("--trajectory needs a workload with several steps and the global selection")
    seed = rank_seeds(gb.rank, 1)[0]
    si = gb.with_budget(syn.make_sequence(wl, seq=0, seed=seed))
    st = sk.init_state(gb.config(1))
    P = sk.sel_rows(st.cfg)
    clocks = ClockSampler(gb.local)
    t0 = time.time()
    rows, tok_sum, ms_sum, e2e_ms_sum, launches = [], 0, 0.0, 0.0, 0
    kt_sum, work_sum = {}, None
    n_kt = max(1, min(args.steps, 20))
    h2d_sum = d2h_sum = 0
    for step in range(wl.steps):
        seq = gb.make_seq(si, 0, P)
        ws = sk.workspace(st, [seq], device=gb.dev)
        work = work_per_step(wl, [dict(L=si.L, B=si.budget)], per_head=P > 1)
        snap = sk.export_slot(st, 0)
        torch.cuda.synchronize(gb.dev)
        ms, nl = gb.time_steps(st, [seq], ws, args.steps, args.warmup)
        launches += nl
        ms = max_over_ranks(ms, gb.dist, gb.dev)
        kt = gb.kernel_pass(st, [seq], ws, n_kt)
        e_ms = None
        if not args.no_e2e:
            sk.import_slot(st, 0, snap)
            e_ms, h2d, d2h = gb.e2e(st, [si], P, 3, [seq])
            e2e_ms_sum += e_ms
            h2d_sum += h2d
            d2h_sum += d2h
        sk.import_slot(st, 0, snap)
        sk.step(st, [seq], ws)   # the step itself, from the restored state
        torch.cuda.synchronize(gb.dev)
        sk.check_device_error(st)
        ms_step = ms / args.steps
        roof, kernels = gb.roofline(kt, work, n_kt, args.workload)
        rows.append({"step": step, "L": si.L, "B": si.budget, "tokens": work["tokens"], "ms": ms_step,
                     "tokens_per_s": work["tokens"] / (ms_step / 1e3),
                     "step_roofline_frac": gb.step_roofline(work, ms_step)["frac"],
                     "roofline_us": gb.step_roofline(work, ms_step)["roofline_us"],
                     "kernels_us": {k: v["avg_us"] for k, v in kernels.items()},
                     "e2e_ms": e_ms})
        tok_sum += work["tokens"]
        ms_sum += ms_step
        for k, v in kt.items():
            a = kt_sum.get(k, (0, 0.0))
            kt_sum[k] = (a[0] + v[0], a[1] + v[1])
        work_sum = work if work_sum is None else {k: work_sum[k] + work[k] for k in work}
        if step + 1 == wl.steps:
            break
        lp = si.L - wl.window
        layouts = [si.layout[l].take(np.concatenate([seq.idx[l, 0].cpu().numpy(), np.arange(lp, si.L)]))
                   for l in range(wl.n_layers)]
        si = gb.with_budget(syn.append_step(wl, seq.k_out.cpu(), seq.v_out.cpu(), layouts, step + 1,
                                            si.n_visual_history, seed=seed))
    t_end = time.time()
    clocks.stop()
    roofline, kernels = gb.roofline(kt_sum, work_sum, n_kt, args.workload)
    step_roofline = gb.step_roofline(work_sum, ms_sum)
    value = job_throughput(tok_sum, gb.world, 1, ms_sum)
    e2e = None
    if not args.no_e2e:
        e2e = {"value": job_throughput(tok_sum, gb.world, 1, e2e_ms_sum), "unit": UNIT,
               "h2d_bytes_per_step": h2d_sum / wl.steps, "d2h_bytes_per_step": d2h_sum / wl.steps,
               "steps": 3, "ms_per_step": e2e_ms_sum / wl.steps}
    cpu = cpu1 = None
    if gb.rank == 0 and gb.world == 1 and not args.no_cpu_baseline:
        cpu, cpu1 = cpu_baselines(args)
    if gb.rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": gb.world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_sum / wl.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": args.workload, "mode": f"trajectory of {wl.steps} steps, each timed on "
                       "its own input (the previous step's GPU compaction plus one screenshot and "
                       f"{wl.step_text} text tokens), state carried",
                       "select_mode": args.select_mode, "layers": wl.n_layers, "w": wl.window,
                       "budget_pct": args.budget_pct or wl.budget_pct,
                       "l2": "inputs 0.5-1.2 GB per step > 129 MB L2 (no flush)",
                       "parallelism": f"replicas x{gb.world}"},
            "trajectory_steps": rows, "step_roofline": step_roofline, "roofline": roofline,
            "kernels": kernels, "cpu_baseline": cpu, "cpu_baseline_1thread": cpu1, "e2e": e2e,
            "gpu_launches": launches, "clocks": clocks.summary(t0, t_end),
        }))
    if gb.dist is not None:
        gb.dist.destroy_process_group()
    st.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["starkv", "reference"], default="starkv")
    ap.add_argument("--workload", default="uitars_5shot_28l")
    ap.add_argument("--select-mode", choices=["global", "per_head"], default="global",
                    help="global top-B per layer (the paper's) or one top-B per KV group")
    ap.add_argument("--lse", choices=["computed", "given"], default="computed",
                    help="given: every step first runs the window-attention producer (the model's "
                         "attention of the window rows) and the compression takes its normalisers, "
                         "so the first scoring pass is skipped")
    ap.add_argument("--budget-pct", type=int, default=0,
                    help="budget as this percentage of the visual tokens (0: the workload's own)")
    ap.add_argument("--trajectory", action="store_true",
                    help="run the workload's steps as a trajectory (config 3), timing each step")
    ap.add_argument("--soak-s", type=float, default=2.0)
    ap.add_argument("--cpu-budget-s", type=float, default=15.0)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--oracle-worker", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--budget-s", type=float, default=15.0, help=argparse.SUPPRESS)
    ap.add_argument("--max-layers", type=int, default=28, help=argparse.SUPPRESS)
    ap.add_argument("--repeat", type=int, default=0, help=argparse.SUPPRESS)
    args = ap.parse_args()
    if args.oracle_worker:
        oracle_worker(args)
    elif args.impl == "reference":
        reference_arm(args)
    else:
        gpu_arm(args)


if __name__ == "__main__":
    main()
