"""Benchmark of the SBD block step on GB300.

One step = one pass of the whole hot path over one batch of synthetic input:
block attention (Eq. 5) -> LM head with fused entropy and Gumbel-max
sampling (Eqs. 6-7) -> EB select (Eq. 3), through the C ABI of libsbd.
The block state (masked flags, block tokens) is restored before every step
so that every step does the same work.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
    python bench.py --impl reference ...   # the fp64 oracle on host cores

Prints one JSON line (rank 0).  Under torchrun every rank runs an
independent replica on its own GPU (the block step does not shard: no data
path collective); the time is the max over ranks.
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import gen  # noqa: E402

METRIC = "us per SBD block step (attention + LM head/entropy/Gumbel + EB select)"
UNIT = "us"
FALLBACK_HBM_GBS = 6800.0


# ------------------------------------------------------------------ helpers

def dist_env():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def max_over_ranks(x: float, world: int, device="cpu") -> float:
    """The largest x over all ranks (a barrier follows); x itself at N = 1.
    The timed region of every replica is reduced this way."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.barrier()
    return float(t.item())


def job_us_per_step(job_ms: float, steps_per_rank: int, world: int) -> float:
    """Whole-job time per step: each of `world` replicas ran `steps_per_rank`
    steps within `job_ms`, the slowest rank's time."""
    return job_ms * 1000.0 / (steps_per_rank * world)


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f), "measured"
    return {"hbm_gbs": FALLBACK_HBM_GBS, "bf16_tflops": 1900.0,
            "bf16_tflops_sustained": 1700.0}, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 100 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,"
              "clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.rows = []
        self.proc = None
        self.marks = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append((time.time(), line.strip()))

    def mark(self, name):
        self.marks.append((name, time.time()))

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=2)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        return self.summary()

    def summary(self):
        marks = dict(self.marks)
        t0 = marks.get("timed_start", 0.0)
        t1 = marks.get("timed_end", time.time())
        parsed = []
        for t, line in self.rows:
            p = [x.strip() for x in line.split(",")]
            if len(p) < 10:
                continue
            try:
                parsed.append(dict(t=t, sm=float(p[1]), smax=float(p[2]), util=float(p[4]),
                                   hw=p[6], hwt=p[7], swt=p[8], pcap=p[9]))
            except ValueError:
                continue
        window = "timed"
        sel = [r for r in parsed if t0 - 0.1 <= r["t"] <= t1 + 0.1]
        if not sel:
            window = "bench process (timed region shorter than the 100 ms sampling period)"
            sel = [r for r in parsed if r["util"] > 0] or parsed
        if not sel:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        reasons = set()
        for r in sel:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("pcap", "sw_power_cap")):
                if r[key].lower() == "active":
                    reasons.add(name)
        loaded = [r["sm"] for r in sel if r["util"] > 0] or [r["sm"] for r in sel]
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(r["smax"] for r in sel),
                "reasons": sorted(reasons), "samples": len(sel), "window": window}


def source_sha(path: str) -> str:
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def profiled_traffic(workload: str, kernel_file: str):
    """DRAM bytes per launch of the dominant kernel from the committed ncu
    summary, only while the kernel source is unchanged since the capture."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        table = json.load(f)
    ent = table.get(workload)
    if not ent:
        return None
    if ent.get("source_sha") != source_sha(kernel_file):
        return None
    return ent.get("dram_bytes_per_launch")


# ------------------------------------------------------------------ inputs

def host_inputs(w: gen.Workload, seed: int):
    d = gen.step_inputs(w, seed, step=0, poison_tail=True)
    return d


def algorithmic_bytes(w: gen.Workload, d, noise: str = "buffer") -> dict:
    """Bytes the method must move per step: the KV cache rows in use, block
    K/V, Q and O once; W, the masked hidden rows, their Gumbel rows (none
    with in-kernel noise) and the outputs once; the EB state.  Logits are
    never written."""
    e = 2 if w.dtype == "bf16" else 4
    B, k, Hq, Hkv, D = w.batch, w.block_k, w.n_q_heads, w.n_kv_heads, w.head_dim
    L = int(np.sum(d["cache_len"]))
    R = int(d["masked"].sum())
    attn = (2 * L * Hkv * D + 2 * B * k * Hkv * D + 2 * B * k * Hq * D) * e + B * 4
    noise_bytes = R * w.vocab * 4 if noise == "buffer" else 0
    head = (w.vocab * w.hidden + R * w.hidden) * e + noise_bytes + B * k * (1 + 8)
    eb = B * k * (4 + 4 + 1 + 4 + 1 + 4) + B * 4
    return {"attention": attn * w.n_layers, "head": head, "eb": eb, "R": R}


# ------------------------------------------------------------------ our arm

def run_ours(args):
    import torch

    import paper_2509_04185_gb300 as sbd

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    w = gen.get_workload(args.workload)
    d = host_inputs(w, args.seed)
    dt = w.dtype

    def to_dev(x):
        x = np.ascontiguousarray(x)
        if dt == "bf16" and x.dtype == np.uint16:
            return torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).to(dev)
        return torch.from_numpy(x).to(dev)

    T = {k: to_dev(d[k]) for k in ("q", "k_cache", "v_cache", "k_blk", "v_blk", "hidden", "w")}
    T["cache_len"] = torch.from_numpy(d["cache_len"]).to(dev)
    T["gumbel"] = torch.from_numpy(d["gumbel"]).to(dev)
    masked0 = torch.from_numpy(d["masked"]).to(dev)
    bt0 = torch.from_numpy(d["block_tokens"]).to(dev)
    masked = masked0.clone()
    bt = bt0.clone()
    out = torch.empty_like(T["q"])
    ent = torch.empty(masked.shape, dtype=torch.float32, device=dev)
    tok = torch.empty(masked.shape, dtype=torch.int32, device=dev)
    n_un = torch.empty(w.batch, dtype=torch.int32, device=dev)
    import ctypes
    ad = sbd.attn_desc(T["q"], T["k_cache"])
    hd = sbd.head_desc(T["hidden"], T["w"])
    ws_a = torch.empty(max(1, sbd.lib.sbd_block_attention_workspace_size(ctypes.byref(ad))),
                       dtype=torch.uint8, device=dev)
    ws_h = torch.empty(max(1, sbd.lib.sbd_head_entropy_sample_workspace_size(ctypes.byref(hd))),
                       dtype=torch.uint8, device=dev)
    # a dedicated stream: the step is captured into a CUDA graph on it
    stream = torch.cuda.Stream(dev)
    gamma, tau = args.gamma, args.tau

    attn_call = sbd.prepare_block_attention(T["q"], T["k_cache"], T["v_cache"], T["cache_len"],
                                            T["k_blk"], T["v_blk"], out, ws_a, stream=stream)
    if args.noise == "philox":
        # in-kernel counter-based noise: no noise tensor is read
        head_call = sbd.prepare_head_entropy_sample_philox(T["hidden"], T["w"], masked, args.seed,
                                                           0, tau, ent, tok, ws_h, stream=stream)
    else:
        head_call = sbd.prepare_head_entropy_sample(T["hidden"], T["w"], masked, T["gumbel"], tau,
                                                    ent, tok, ws_h, stream=stream)
    step_inputs = ("q", "k_blk", "v_blk", "hidden") + (("gumbel",) if args.noise == "buffer" else ())
    eb_call = sbd.prepare_eb_select(ent, tok, gamma, masked, bt, n_un, stream=stream)

    # The restore of the block state before each step (so that every timed
    # step starts from the same masked positions) is harness, not method:
    # it runs on a side stream beside the attention, which reads neither,
    # and the LM head waits for it.
    restore_stream = torch.cuda.Stream(dev)

    def step(ev=None):
        with torch.cuda.stream(stream):
            fork = torch.cuda.Event()
            fork.record(stream)
            restore_stream.wait_event(fork)
            with torch.cuda.stream(restore_stream):
                masked.copy_(masked0, non_blocking=True)
                bt.copy_(bt0, non_blocking=True)
            restored = torch.cuda.Event()
            restored.record(restore_stream)
            if ev is not None:
                ev[0].record(stream)
            attn_call()
            if ev is not None:
                ev[1].record(stream)
            stream.wait_event(restored)
            head_call()
            if ev is not None:
                ev[2].record(stream)
            eb_call()
            if ev is not None:
                ev[3].record(stream)

    torch.cuda.synchronize(dev)        # inputs were made on the default stream
    sampler = ClockSampler(local_rank) if rank == 0 else None
    if sampler:
        sampler.start()
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    if sbd.sbd_device_error() != 0:
        raise RuntimeError("device error word set during warm-up")

    # The whole step (state restore + three library calls, 6-7 kernels with
    # programmatic dependent launch between them) captured once as a graph.
    graph = None
    if not args.no_graph:
        try:
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph, stream=stream):
                step()
            for _ in range(3):
                with torch.cuda.stream(stream):
                    graph.replay()
            torch.cuda.synchronize(dev)
        except Exception as ex:  # capture unsupported here: time the eager step
            print(f"graph capture failed ({ex}); timing eager steps", file=sys.stderr)
            graph = None

    # ---- timed region: K steps, events on the launching stream
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    if sampler:
        sampler.mark("timed_start")
    start.record(stream)
    with torch.cuda.stream(stream):
        for i in range(args.steps):
            if graph is not None:
                graph.replay()
            else:
                step()
    end.record(stream)
    torch.cuda.synchronize(dev)
    if sampler:
        sampler.mark("timed_end")
    total_ms = max_over_ranks(start.elapsed_time(end), world, dev)
    n_accepted = int(n_un.sum().item())
    if sbd.sbd_device_error() != 0:
        raise RuntimeError("device error word set during the timed region")

    # ---- per-call durations (eager steps, events between the calls on the
    # launching stream): the roofline of the dominant kernel
    n_ev = max(1, min(args.steps, 500))
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_ev)]
    for i in range(n_ev):
        step(evs[i])
    torch.cuda.synchronize(dev)
    attn_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    head_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
    eb_ms = statistics.mean(e[2].elapsed_time(e[3]) for e in evs)

    # ---- end to end through host buffers (pinned), copies inside the region.
    # Two sets of device inputs and results: while step s runs on the
    # compute stream, the inputs of step s + 1 are copied up on a second
    # stream, into the other set, and step s - 1's results are read back on
    # a third.  Every step's copies are inside the timed region.
    e2e = None
    if not args.skip_e2e:
        host = {}
        for k in step_inputs:
            host[k] = torch.empty_like(T[k], device="cpu").pin_memory()
            host[k].copy_(T[k])
        host["masked"] = masked0.cpu().pin_memory()
        host["block_tokens"] = bt0.cpu().pin_memory()
        res_names = ("out", "ent", "tok", "masked", "bt", "n_un")
        sets = []
        for _ in range(2):
            S = {k: torch.empty_like(T[k]) for k in step_inputs}
            S.update(masked=torch.empty_like(masked), bt=torch.empty_like(bt),
                     out=torch.empty_like(out), ent=torch.empty_like(ent),
                     tok=torch.empty_like(tok), n_un=torch.empty_like(n_un))
            calls = [sbd.prepare_block_attention(S["q"], T["k_cache"], T["v_cache"],
                                                 T["cache_len"], S["k_blk"], S["v_blk"], S["out"],
                                                 ws_a, stream=stream)]
            if args.noise == "philox":
                calls.append(sbd.prepare_head_entropy_sample_philox(
                    S["hidden"], T["w"], S["masked"], args.seed, 0, tau, S["ent"], S["tok"], ws_h,
                    stream=stream))
            else:
                calls.append(sbd.prepare_head_entropy_sample(
                    S["hidden"], T["w"], S["masked"], S["gumbel"], tau, S["ent"], S["tok"], ws_h,
                    stream=stream))
            calls.append(sbd.prepare_eb_select(S["ent"], S["tok"], gamma, S["masked"], S["bt"],
                                               S["n_un"], stream=stream))
            S["calls"] = calls
            S["res"] = {k: torch.empty_like(S[k], device="cpu").pin_memory() for k in res_names}
            sets.append(S)
        h2d = sum(v.numel() * v.element_size() for v in host.values())
        d2h = sum(v.numel() * v.element_size() for v in sets[0]["res"].values())
        n_e2e = max(1, min(args.steps, 200))
        copy_stream = torch.cuda.Stream(dev)         # host -> device
        back_stream = torch.cuda.Stream(dev)         # device -> host
        uploaded = [torch.cuda.Event() for _ in range(2)]
        released = [torch.cuda.Event() for _ in range(2)]

        def upload(i):
            S = sets[i]
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(released[i])      # the set's previous step is done
                for k in step_inputs:
                    S[k].copy_(host[k], non_blocking=True)
                S["masked"].copy_(host["masked"], non_blocking=True)
                S["bt"].copy_(host["block_tokens"], non_blocking=True)
                uploaded[i].record(copy_stream)

        computed = [torch.cuda.Event() for _ in range(2)]

        def calls(S):
            for c in S["calls"]:
                c()

        graphs = [None, None]

        def run(i):
            # the step on the compute stream; its results read back on a
            # third stream, overlapping the next step
            S = sets[i]
            with torch.cuda.stream(stream):
                stream.wait_event(uploaded[i])
                if graphs[i] is not None:
                    graphs[i].replay()
                else:
                    calls(S)
                computed[i].record(stream)
            with torch.cuda.stream(back_stream):
                back_stream.wait_event(computed[i])
                for k in res_names:
                    S["res"][k].copy_(S[k], non_blocking=True)
                released[i].record(back_stream)

        def e2e_steps(n, start_ev=None):
            if start_ev is not None:
                copy_stream.wait_event(start_ev)
            upload(0)
            for s_ in range(n):
                if s_ + 1 < n:
                    upload((s_ + 1) % 2)
                run(s_ % 2)
            stream.wait_event(released[(n - 1) % 2])     # the last readback is in

        e2e_steps(3)
        torch.cuda.synchronize(dev)
        if not args.no_graph:
            # each set's calls as one graph, as in the device timing
            for i in range(2):
                graphs[i] = torch.cuda.CUDAGraph()
                with torch.cuda.graph(graphs[i], stream=stream):
                    calls(sets[i])
            e2e_steps(3)
            torch.cuda.synchronize(dev)
        s2 = torch.cuda.Event(enable_timing=True)
        e2 = torch.cuda.Event(enable_timing=True)
        s2.record(stream)
        e2e_steps(n_e2e, s2)
        e2.record(stream)
        torch.cuda.synchronize(dev)
        if sbd.sbd_device_error() != 0:
            raise RuntimeError("device error word set during the end-to-end steps")
        # every step had the same inputs: the last step read back must match
        # the device-timed steps' results
        last = sets[(n_e2e - 1) % 2]["res"]
        for k_, ref_ in (("tok", tok), ("n_un", n_un), ("masked", masked), ("bt", bt)):
            if not torch.equal(last[k_], ref_.cpu()):
                raise RuntimeError(f"end-to-end step read back a different {k_}")
        e2e_ms = max_over_ranks(s2.elapsed_time(e2), world, dev) / n_e2e
        e2e = {"value": round(job_us_per_step(e2e_ms, 1, world), 3), "unit": UNIT,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "steps": n_e2e,
               "pipeline": "two buffer sets: while step s runs, other streams copy up the "
                           "inputs of step s+1 and read back the results of step s-1"}

    clocks = sampler.stop() if sampler else None

    if rank != 0:
        return
    ab = algorithmic_bytes(w, d, args.noise)
    peaks, peak_src = measured_peaks()
    head_bytes = ab["head"]
    achieved = head_bytes / (head_ms * 1e-3) / 1e9
    kernel_file = os.path.join(ROOT, "paper_2509_04185_gb300", "csrc", "lm_head.cu")
    # the committed captures read the noise from a buffer: no figure for the
    # in-kernel noise variant
    traffic = profiled_traffic(args.workload, kernel_file) if args.noise == "buffer" else None
    attn_gbs = ab["attention"] / (attn_ms * 1e-3) / 1e9
    step_bytes = ab["attention"] + ab["head"] + ab["eb"]
    ms_per_step = total_ms / args.steps
    value_us = job_us_per_step(total_ms, args.steps, world)
    cpu = None
    if world == 1 and not args.skip_cpu:
        cpu = cpu_baseline(w, d, args)

    line = {
        "metric": METRIC,
        "value": round(value_us, 3),
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 6),
        "higher_is_better": False,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16" if dt == "bf16" else "f32",
        "data": "synthetic (seeded generator, shapes of the workload; random-init LM head)",
        "config": {
            "workload": args.workload, "batch": w.batch, "block_k": w.block_k,
            "n_q_heads": w.n_q_heads, "n_kv_heads": w.n_kv_heads, "head_dim": w.head_dim,
            "cache_len": w.cache_len if not isinstance(w.cache_len, tuple) else list(w.cache_len),
            "hidden": w.hidden, "vocab": w.vocab, "masked_rows": ab["R"], "gamma": gamma,
            "tau": tau, "noise": args.noise, "parallelism": f"replicas{world}",
            "l2": "inputs larger than L2: the 1.05 GB+ LM-head weight is streamed every step",
        },
        "gpu_launches": int(args.steps * launches_per_step(sbd, T, ws_a)),
        "per_call_us": {"attention": round(attn_ms * 1000, 3), "head": round(head_ms * 1000, 3),
                        "eb_select": round(eb_ms * 1000, 3)},
        "step_hbm_gbs": round(step_bytes / (ms_per_step * 1e-3) / 1e9, 1),
        "attention_hbm_gbs": round(attn_gbs, 1),
        "tokens_committed_per_s": round(n_accepted / (ms_per_step * 1e-3) * world, 1),
        "roofline": {
            "kernel": "LM head call (compact_rows + head_tc_kernel or head_pair_kernel, tcgen05 + head_combine)",
            "bound": "hbm", "achieved": round(achieved, 1),
            "peak": peaks["hbm_gbs"], "peak_source": peak_src, "unit": "GB/s",
            "frac": round(achieved / peaks["hbm_gbs"], 4),
            "traffic": traffic, "algorithmic_bytes": int(head_bytes),
        },
        "clocks": clocks,
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    print(json.dumps(line), flush=True)


def launches_per_step(sbd, T, ws_a) -> int:
    """Kernels of libsbd per step: attention (+ split combine), compaction,
    LM head, head combine, EB select."""
    import ctypes
    ad = sbd.attn_desc(T["q"], T["k_cache"])
    split = sbd.lib.sbd_block_attention_workspace_size(ctypes.byref(ad)) > 0
    return (2 if split else 1) + 3 + 1


# ------------------------------------------------------------------ oracle

def _oracle_step(w, d, hkv_heads, vocab_rows, gamma, tau):
    """The oracle on a sample of one step: attention for the query heads of
    `hkv_heads` KV heads, the LM head over the first `vocab_rows` vocabulary
    rows of every masked position, then the EB select of the batch."""
    import oracle
    dt = w.dtype
    G = w.n_q_heads // w.n_kv_heads
    q = oracle.widen(d["q"][:, :, : hkv_heads * G], dt)
    kc = oracle.widen(d["k_cache"][:, :, :hkv_heads], dt)
    vc = oracle.widen(d["v_cache"][:, :, :hkv_heads], dt)
    kb = oracle.widen(d["k_blk"][:, :, :hkv_heads], dt)
    vb = oracle.widen(d["v_blk"][:, :, :hkv_heads], dt)
    oracle.block_attention(q, kc, vc, d["cache_len"], kb, vb)
    ent, tok, _ = oracle.head_entropy_sample(oracle.widen(d["hidden"], dt), d["w"][:vocab_rows],
                                             dt, d["masked"], d["gumbel"][:, :, :vocab_rows], tau)
    oracle.eb_select(ent, tok, d["masked"], d["block_tokens"], gamma)


def cpu_baseline(w, d, args, target_s: float = 15.0):
    """Times the oracle (as it stands) on the host cores on a bounded sample
    of the step, scaled to a full step: a fraction 1/f of the KV heads and
    of the vocabulary.  f is the smallest power of two whose sample runs in
    about target_s seconds (measured by a small calibration sample)."""
    f = w.n_kv_heads
    while f > 1 and w.vocab // f < 512:
        f //= 2
    t0 = time.perf_counter()
    _oracle_step(w, d, max(1, w.n_kv_heads // f), w.vocab // f, args.gamma, args.tau)
    t_cal = time.perf_counter() - t0
    frac = 1.0 / f
    while frac < 1.0 and t_cal * 2 < target_s:
        frac *= 2
        t_cal *= 2
    hkv = max(1, int(round(w.n_kv_heads * frac)))
    vrows = max(1, int(round(w.vocab * frac)))
    t0 = time.perf_counter()
    _oracle_step(w, d, hkv, vrows, args.gamma, args.tau)
    dt = time.perf_counter() - t0
    scale = 0.5 * (w.n_kv_heads / hkv) + 0.5 * (w.vocab / vrows)
    return {"value": round(dt * scale * 1e6, 1), "unit": UNIT, "cores": os.cpu_count(),
            "kind": "oracle",
            "sample": (f"fp64 numpy oracle on {hkv}/{w.n_kv_heads} KV heads and {vrows}/{w.vocab} "
                       f"vocab rows of one {w.name} step ({dt:.2f} s), scaled to a full step; "
                       f"BLAS threads = all host cores")}


def run_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return
    w = gen.get_workload(args.workload)
    d = host_inputs(w, args.seed)
    # per-step sample sized so that warmup + steps end within about 2 minutes
    budget = 120.0 / max(1, args.steps + args.warmup)
    f = w.n_kv_heads
    while f > 1 and w.vocab // f < 512:
        f //= 2
    hkv = max(1, w.n_kv_heads // f)
    vrows = w.vocab // f
    t0 = time.perf_counter()
    _oracle_step(w, d, hkv, vrows, args.gamma, args.tau)
    t_cal = time.perf_counter() - t0
    frac = 1.0 / f
    while frac < 1.0 and t_cal * 2 < budget:
        frac *= 2
        t_cal *= 2
    hkv = max(1, int(round(w.n_kv_heads * frac)))
    vrows = max(1, int(round(w.vocab * frac)))
    for _ in range(args.warmup):
        _oracle_step(w, d, hkv, vrows, args.gamma, args.tau)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        _oracle_step(w, d, hkv, vrows, args.gamma, args.tau)
        times.append(time.perf_counter() - t0)
    scale = 0.5 * (w.n_kv_heads / hkv) + 0.5 * (w.vocab / vrows)
    step_s = statistics.mean(times) * scale
    value = round(step_s * 1e6, 1)
    sample = (f"fp64 numpy oracle on {hkv}/{w.n_kv_heads} KV heads and {vrows}/{w.vocab} vocab rows "
              f"of one {w.name} step per timed step, scaled to a full step")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(step_s * 1e3, 3),
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic (seeded generator)",
        "config": {"workload": args.workload, "batch": w.batch, "block_k": w.block_k,
                   "vocab": w.vocab, "hidden": w.hidden, "gamma": args.gamma, "tau": args.tau},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ sweep

class SweepLoop:
    """Device state and prepared ABI calls of the block-step loop of
    Algorithm 3 over an n_layers-layer model: every block starts fully
    masked; each step runs block attention over every layer's KV cache, the
    LM head with entropy and Gumbel-max sampling over the still-masked
    positions, and the EB select; steps repeat until no position of any
    sequence is masked (one 4-byte read of the remaining count per step).

    The per-layer caches and the other large inputs are drawn on the device
    with PyTorch's seeded generator.  Hidden rows are drawn per step of a
    block (hidden[s] feeds step s); the Gumbel noise of a block is drawn
    once and indexed by block position, so each committed token is a
    Gumbel-max sample at its commit step.  With noise="philox" the LM-head
    kernel generates the noise itself, with counter offset s at step s."""

    def __init__(self, w: "gen.Workload", seed: int, noise: str, tau: float, gamma: float,
                 dev, stream):
        import ctypes

        import torch

        import paper_2509_04185_gb300 as sbd
        self.sbd, self.w, self.stream = sbd, w, stream
        self.noise, self.tau, self.gamma, self.seed = noise, tau, gamma, seed
        B, k, Hq, Hkv, D, L = (w.batch, w.block_k, w.n_q_heads, w.n_kv_heads, w.head_dim,
                               w.max_cache_len)
        V, H, NL = w.vocab, w.hidden, w.n_layers
        g = torch.Generator(device=dev)
        g.manual_seed(seed * 1000003 + 17)

        def randn(*shape, std=1.0):
            return (torch.randn(*shape, generator=g, device=dev, dtype=torch.float32)
                    * std).bfloat16()

        self.layers = []
        for _ in range(NL):
            self.layers.append(dict(q=randn(B, k, Hq, D), kc=randn(B, L, Hkv, D),
                                    vc=randn(B, L, Hkv, D), kb=randn(B, k, Hkv, D),
                                    vb=randn(B, k, Hkv, D)))
        self.lens = torch.full((B,), L, dtype=torch.int32, device=dev)
        self.W = randn(V, H, std=w.w_std)
        lo, hi = np.log(w.hidden_scale[0]), np.log(w.hidden_scale[1])
        self.hidden = []
        for _ in range(k):
            h = torch.randn(B, k, H, generator=g, device=dev)
            sc = torch.exp(torch.empty(B, k, 1, device=dev).uniform_(lo, hi, generator=g))
            self.hidden.append((h * sc).bfloat16())
        u = torch.rand(B, k, V, generator=g, device=dev, dtype=torch.float64).clamp_(
            1e-300, 1 - 1e-16)
        self.gumbel = (-torch.log(-torch.log(u))).float()
        del u
        self.outs = [torch.empty_like(self.layers[0]["q"]) for _ in range(NL)]
        self.masked = torch.ones(B, k, dtype=torch.uint8, device=dev)
        self.bt = torch.full((B, k), -1, dtype=torch.int32, device=dev)
        self.ent = torch.empty(B, k, dtype=torch.float32, device=dev)
        self.tok = torch.empty(B, k, dtype=torch.int32, device=dev)
        self.n_un = torch.empty(B, dtype=torch.int32, device=dev)
        self.left_h = torch.empty(1, dtype=torch.int32).pin_memory()
        ad = sbd.attn_desc(self.layers[0]["q"], self.layers[0]["kc"])
        self.ws_a = torch.empty(max(1, sbd.lib.sbd_block_attention_workspace_size(
            ctypes.byref(ad))), dtype=torch.uint8, device=dev)
        hd = sbd.head_desc(self.hidden[0], self.W)
        self.ws_h = torch.empty(max(1, sbd.lib.sbd_head_entropy_sample_workspace_size(
            ctypes.byref(hd))), dtype=torch.uint8, device=dev)
        self.attn_calls = [
            sbd.prepare_block_attention(L_["q"], L_["kc"], L_["vc"], self.lens, L_["kb"],
                                        L_["vb"], self.outs[i], self.ws_a, stream=stream)
            for i, L_ in enumerate(self.layers)]
        if noise == "philox":
            self.head_calls = [
                sbd.prepare_head_entropy_sample_philox(self.hidden[s_], self.W, self.masked, seed,
                                                       s_, tau, self.ent, self.tok, self.ws_h,
                                                       stream=stream)
                for s_ in range(k)]
        else:
            self.head_calls = [
                sbd.prepare_head_entropy_sample(self.hidden[s_], self.W, self.masked, self.gumbel,
                                                tau, self.ent, self.tok, self.ws_h, stream=stream)
                for s_ in range(k)]
        self.eb_call = sbd.prepare_eb_select(self.ent, self.tok, gamma, self.masked, self.bt,
                                             self.n_un, stream=stream)
        self.graphs = []

    def _graph_step(self, s_: int) -> None:
        import torch
        for c in self.attn_calls:
            c()
        self.head_calls[s_]()
        self.eb_call()
        self.left_h.copy_(self.masked.sum(dtype=torch.int32).view(1), non_blocking=True)

    def capture(self) -> None:
        """One CUDA graph per step index s = 0 .. k-1: every layer's
        attention, the LM head of step s, the EB select and the 4-byte read
        of the remaining masked count into pinned host memory.  block() then
        launches one graph per step instead of each kernel from the host.
        The loop's stream must not be the legacy default stream."""
        import torch
        graphs = []
        with torch.cuda.stream(self.stream):
            for s_ in range(self.w.block_k):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=self.stream):
                    self._graph_step(s_)
                graphs.append(g)
        self.graphs = graphs

    def launches_per_step(self) -> int:
        """Kernels one step launches: per layer the attention kernel (+ the
        split combine when the workspace is in use), the head's compaction,
        main and combine kernels, and the EB select."""
        return self.w.n_layers * (2 if self.ws_a.numel() > 1 else 1) + 3 + 1

    def block(self, ev=None, trace=None) -> int:
        """One block: steps until no masks.  Returns the step count.  ev:
        a list that gets four CUDA events per step (start, after attention,
        after the head, after EB).  trace: a list that gets, per step, host
        copies of the block state before and after the step and of the
        head's outputs (this adds synchronisation; tests only)."""
        import torch
        k = self.w.block_k
        stream = self.stream
        graphed = bool(self.graphs) and ev is None and trace is None
        with torch.cuda.stream(stream):
            return self._block(k, stream, graphed, ev, trace)

    def _block(self, k, stream, graphed, ev, trace) -> int:
        import torch
        self.masked.fill_(1)
        self.bt.fill_(-1)
        steps = 0
        while True:
            if graphed:
                self.graphs[min(steps, k - 1)].replay()
                stream.synchronize()
                steps += 1
                if int(self.left_h.item()) == 0 or steps >= k:
                    return steps
                continue
            if trace is not None:
                stream.synchronize()
                before = (self.masked.cpu().numpy(), self.bt.cpu().numpy())
            if ev is not None:
                ev.append([torch.cuda.Event(enable_timing=True) for _ in range(4)])
                ev[-1][0].record(stream)
            for c in self.attn_calls:
                c()
            if ev is not None:
                ev[-1][1].record(stream)
            self.head_calls[min(steps, k - 1)]()
            if ev is not None:
                ev[-1][2].record(stream)
            self.eb_call()
            if ev is not None:
                ev[-1][3].record(stream)
            self.left_h.copy_(self.masked.sum(dtype=torch.int32).view(1), non_blocking=True)
            stream.synchronize()
            if trace is not None:
                trace.append(dict(step=steps, masked_before=before[0], bt_before=before[1],
                                  entropy=self.ent.cpu().numpy(), token=self.tok.cpu().numpy(),
                                  masked_after=self.masked.cpu().numpy(),
                                  bt_after=self.bt.cpu().numpy(),
                                  n_unmasked=self.n_un.cpu().numpy()))
            steps += 1
            if int(self.left_h.item()) == 0 or steps >= k:
                return steps


def run_sweep(args):
    """The 32-layer block-step loop at Llama-3.1-8B attention shapes
    (Algorithm 3), driven by SweepLoop.  A timed step is one iteration of
    the loop; the timed region covers whole blocks."""
    import torch

    import paper_2509_04185_gb300 as sbd

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    w = gen.get_workload(args.workload)
    B, k, Hq, Hkv, D, L = w.batch, w.block_k, w.n_q_heads, w.n_kv_heads, w.head_dim, w.max_cache_len
    V, H, NL = w.vocab, w.hidden, w.n_layers
    # a stream of its own: each step is replayed as a CUDA graph on it
    stream = torch.cuda.Stream(dev)
    torch.cuda.synchronize(dev)
    loop = SweepLoop(w, args.seed, args.noise, args.tau, args.gamma, dev, stream)
    torch.cuda.synchronize(dev)
    block = loop.block

    sampler = ClockSampler(local_rank) if rank == 0 else None
    if sampler:
        sampler.start()
    n_warm = max(1, args.warmup // max(1, k // 2))
    for _ in range(n_warm):
        block()
    torch.cuda.synchronize(dev)
    graphed = False
    if not args.no_graph:
        try:
            loop.capture()
            block()
            torch.cuda.synchronize(dev)
            graphed = True
        except Exception as ex:  # capture unsupported here: time the eager loop
            print(f"sweep graph capture failed ({ex}); timing eager steps", file=sys.stderr)
            loop.graphs = []
    if sbd.sbd_device_error() != 0:
        raise RuntimeError("device error word set during warm-up")
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    if sampler:
        sampler.mark("timed_start")
    t0 = time.perf_counter()
    n_steps, n_blocks = 0, 0
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    while n_steps < args.steps:
        n_steps += block()
        n_blocks += 1
    end.record(stream)
    torch.cuda.synchronize(dev)
    wall = time.perf_counter() - t0
    if sampler:
        sampler.mark("timed_end")
    total_ms = max_over_ranks(start.elapsed_time(end), world, dev)
    # per-call durations: eager blocks with events between the calls, after
    # the timed region
    evs = []
    for _ in range(2):
        block(evs)
    torch.cuda.synchronize(dev)
    attn_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    head_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
    eb_ms = statistics.mean(e[2].elapsed_time(e[3]) for e in evs)
    if sbd.sbd_device_error() != 0:
        raise RuntimeError("device error word set during the timed region")
    clocks = sampler.stop() if sampler else None
    if rank != 0:
        return
    peaks, peak_src = measured_peaks()
    e = 2
    attn_bytes = NL * (2 * B * L * Hkv * D + 2 * B * k * Hkv * D + 2 * B * k * Hq * D) * e
    # masked rows average over the steps of a block: k rows at the first step
    head_bytes_first = V * H * e + B * k * H * e + (B * k * V * 4 if args.noise == "buffer" else 0)
    ms_per_step = total_ms / n_steps
    attn_gbs = attn_bytes / (attn_ms * 1e-3) / 1e9
    # DRAM bytes of one layer's attention launch from the committed capture
    # (while the kernel source is unchanged), times the layers of a step
    per_launch = profiled_traffic(args.workload, os.path.join(
        ROOT, "paper_2509_04185_gb300", "csrc", "block_attention_tc.cu"))
    sweep_traffic = int(per_launch * NL) if per_launch else None
    line = {
        "metric": METRIC, "value": round(job_us_per_step(total_ms, n_steps, world), 3), "unit": UNIT,
        "n_gpus": world, "steps": n_steps, "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 6), "higher_is_better": False, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (PyTorch seeded device generator; random-init LM head)",
        "config": {"workload": args.workload, "batch": B, "block_k": k, "layers": NL,
                   "cache_len": L, "hidden": H, "vocab": V, "gamma": args.gamma, "tau": args.tau,
                   "noise": args.noise,
                   "parallelism": f"replicas{world}",
                   "l2": "inputs larger than L2: 17 GB of KV caches per step"},
        "steps_per_block": round(n_steps / n_blocks, 3),
        "blocks": n_blocks,
        "tokens_committed_per_s": round(n_blocks * B * k / (total_ms * 1e-3) * world, 1),
        "gpu_launches": int(n_steps * loop.launches_per_step()),
        "per_call_us": {"attention_32_layers": round(attn_ms * 1000, 3),
                        "head": round(head_ms * 1000, 3), "eb_select": round(eb_ms * 1000, 3)},
        "roofline": {
            "kernel": "block attention, 32 layers (attn_tc_kernel up to 64 packed rows, "
                      "attn_wide_kernel above)",
            "bound": "hbm", "achieved": round(attn_gbs, 1), "peak": peaks["hbm_gbs"],
            "peak_source": peak_src, "unit": "GB/s", "frac": round(attn_gbs / peaks["hbm_gbs"], 4),
            "traffic": sweep_traffic, "algorithmic_bytes": int(attn_bytes)},
        "head_first_step_bytes": int(head_bytes_first),
        "host_wall_s": round(wall, 3),
        "step_launch": "one CUDA graph per step (every layer's attention, the LM head, the EB "
                       "select, the 4-byte read of the remaining count)" if graphed
                       else "eager launches",
        "clocks": clocks, "e2e": None, "cpu_baseline": None,
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------- measured speedup tables

SPEEDUP_BATCHES = (1, 4, 16)
SPEEDUP_KV_LENS = (1024, 8192, 32768)
SPEEDUP_KS = (4, 8, 16)
SPEEDUP_NFE = (2, 4)


def run_speedup_tables(args):
    """GB300 wall-clock counterpart of the paper's theoretical speedup tables
    (Sec. "Timing analysis"): time(n) of a full forward of a Llama-3.1-8B-
    shaped model (32 layers, 32/8 heads of 128, hidden 4096, MLP 14336, vocab
    128256, bf16) for a block of n tokens per sequence, measured for n = 1
    (NTP), k, and 2k (the first forward of a block, which also carries the
    previous block's k tokens), then
        slowdown(n)    = time(n) / time(1),
        speedup(l, k)  = k time(1) / (time(2k) + (l - 1) time(k)),  l = k / NFE.
    Per layer (pre-norm, RMSNorm without gain): the fused QKV projection,
    block attention (sbd_block_attention, or sbd_block_attention_causal_prefix
    with the first k rows causal for 2k), the output projection and the
    SiLU-gated MLP; then the final norm and the LM head with entropy and
    Gumbel-max sample (sbd_head_entropy_sample) over the B n rows.
    The projections are the GEMMs of the timing model: plain bf16 GEMMs by
    cuBLAS (torch.matmul), or with --linear sbd by sbd_linear (the LM-head
    kernel with a storing epilogue); the model's linear layers, outside the
    SBD step.  Every layer has its own
    weights and KV cache, so nothing stays in L2 between layers; each forward
    is one CUDA graph, timed with CUDA events over `--steps` replays."""
    import torch

    import paper_2509_04185_gb300 as sbd

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    NL, H, F, V, Hq, Hkv, D = 32, 4096, 14336, 128256, 32, 8, 128
    g = torch.Generator(device=dev)
    g.manual_seed(args.seed * 7919 + 3)

    def randn(*shape, std=1.0):
        return (torch.randn(*shape, generator=g, device=dev, dtype=torch.float32) * std).bfloat16()

    w_std = 0.02
    layers_w = [dict(qkv=randn((Hq + 2 * Hkv) * D, H, std=w_std), o=randn(H, Hq * D, std=w_std),
                     gu=randn(2 * F, H, std=w_std), down=randn(H, F, std=w_std)) for _ in range(NL)]
    w_head = randn(V, H, std=w_std)
    stream = torch.cuda.Stream(dev)
    max_n = 2 * max(SPEEDUP_KS)
    results = []
    sampler = ClockSampler(local_rank) if rank == 0 else None
    if sampler:
        sampler.start()
    for B in SPEEDUP_BATCHES:
        for L in SPEEDUP_KV_LENS:
            if B * max_n > 512:
                continue
            Lmax = L + max_n
            caches = [(randn(B, Lmax, Hkv, D), randn(B, Lmax, Hkv, D)) for _ in range(NL)]
            print(f"speedup tables: batch {B} kv {L}: caches ready", file=sys.stderr, flush=True)
            lens = torch.full((B,), L, dtype=torch.int32, device=dev)
            # (block rows, causal prefix rows): NTP, the block steps, and the
            # first forward of each block size
            forwards = [(1, 0)] + [(k, 0) for k in SPEEDUP_KS] + [(2 * k, k) for k in SPEEDUP_KS]
            times = {}
            for n, n_causal in forwards:
                T = B * n
                x0 = randn(T, H)
                attn_out = torch.empty(B, n, Hq, D, dtype=torch.bfloat16, device=dev)
                ad = sbd.AttnDesc(B, n, Hq, Hkv, D, Lmax, sbd.SBD_DTYPE_BF16, 0.0, 0)
                import ctypes
                ws_a = torch.empty(max(1, sbd.lib.sbd_block_attention_workspace_size(ctypes.byref(ad))),
                                   dtype=torch.uint8, device=dev)
                hid = torch.empty(B, n, H, dtype=torch.bfloat16, device=dev)
                masked = torch.ones(B, n, dtype=torch.uint8, device=dev)
                gum = torch.rand(B, n, V, generator=g, device=dev)
                ent = torch.empty(B, n, device=dev)
                tok = torch.empty(B, n, dtype=torch.int32, device=dev)
                hd = sbd.HeadDesc(B, n, H, V, sbd.SBD_DTYPE_BF16)
                ws_h = torch.empty(sbd.lib.sbd_head_entropy_sample_workspace_size(ctypes.byref(hd)),
                                   dtype=torch.uint8, device=dev)
                qkv_buf = torch.empty(T, (Hq + 2 * Hkv) * D, dtype=torch.bfloat16, device=dev)
                q_v = qkv_buf[:, :Hq * D].view(B, n, Hq, D)
                k_v = qkv_buf[:, Hq * D:(Hq + Hkv) * D]
                v_v = qkv_buf[:, (Hq + Hkv) * D:]
                kb = torch.empty(B, n, Hkv, D, dtype=torch.bfloat16, device=dev)
                vb = torch.empty(B, n, Hkv, D, dtype=torch.bfloat16, device=dev)
                qc = torch.empty(B, n, Hq, D, dtype=torch.bfloat16, device=dev)
                calls = []
                for li in range(NL):
                    kc, vc = caches[li]
                    if n_causal:
                        calls.append(lambda kc=kc, vc=vc: sbd.sbd_block_attention_causal_prefix(
                            qc, kc, vc, lens, kb, vb, n_causal, out=attn_out, workspace=ws_a,
                            stream=stream))
                    else:
                        calls.append(lambda kc=kc, vc=vc: sbd.sbd_block_attention(
                            qc, kc, vc, lens, kb, vb, out=attn_out, workspace=ws_a, stream=stream))

                def linear(x_, w_, out_=None):
                    # the layer's GEMM: cuBLAS (torch.matmul) or sbd_linear
                    if args.linear == "sbd":
                        return sbd.sbd_linear(x_, w_, out=out_, stream=stream)
                    if out_ is None:
                        return torch.matmul(x_, w_.t())
                    return torch.matmul(x_, w_.t(), out=out_)

                def rms(x):
                    xf = x.float()
                    return (xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + 1e-5)).bfloat16()

                def forward():
                    with torch.cuda.stream(stream):
                        x = x0
                        for li in range(NL):
                            Wl = layers_w[li]
                            linear(rms(x), Wl["qkv"], qkv_buf)
                            qc.copy_(q_v)                          # contiguous per-call layouts
                            kb.copy_(k_v.view(B, n, Hkv, D))
                            vb.copy_(v_v.view(B, n, Hkv, D))
                            calls[li]()
                            o = linear(attn_out.view(T, Hq * D), Wl["o"])
                            x = x + o
                            gu = linear(rms(x), Wl["gu"])
                            act = torch.nn.functional.silu(gu[:, :F]) * gu[:, F:]
                            x = x + linear(act, Wl["down"])
                        hid.copy_(rms(x).view(B, n, H))
                        sbd.sbd_head_entropy_sample(hid, w_head, masked, gum, 1.0, ent, tok,
                                                    workspace=ws_h, stream=stream)

                # the inputs above were made on the default stream
                torch.cuda.synchronize(dev)
                for _ in range(3):
                    forward()
                torch.cuda.synchronize(dev)
                graph = torch.cuda.CUDAGraph()
                with torch.cuda.graph(graph, stream=stream):
                    forward()
                for _ in range(max(3, args.warmup)):
                    graph.replay()
                torch.cuda.synchronize(dev)
                reps = max(5, min(args.steps, 50))
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                with torch.cuda.stream(stream):
                    for _ in range(reps):
                        graph.replay()
                e1.record(stream)
                torch.cuda.synchronize(dev)
                times[(n, n_causal)] = e0.elapsed_time(e1) / reps
                if not bool(torch.isfinite(ent).all()):
                    raise RuntimeError(f"non-finite entropy at batch {B} kv {L} block {n}")
                del graph
                print(f"speedup tables: batch {B} kv {L} block {n} (causal {n_causal}): "
                      f"{times[(n, n_causal)]:.3f} ms", file=sys.stderr, flush=True)
            code = sbd.sbd_device_error()
            if code != 0:
                raise RuntimeError(f"device error word {code} at batch {B} kv {L}")
            t1 = times[(1, 0)]
            name = lambda n, c: f"{n}" if c == 0 else f"{n}_first"
            row = {"batch": B, "kv_len": L,
                   "ms_per_forward": {name(n, c): round(t, 4) for (n, c), t in times.items()},
                   "slowdown": {name(n, c): round(t / t1, 4) for (n, c), t in times.items()},
                   "speedup": {}}
            for k in SPEEDUP_KS:
                for nfe in SPEEDUP_NFE:
                    l = k // nfe
                    if l < 1:
                        continue
                    row["speedup"][f"k{k}_nfe{nfe}"] = round(
                        k * t1 / (times[(2 * k, k)] + (l - 1) * times[(k, 0)]), 4)
            results.append(row)
            del caches
            torch.cuda.empty_cache()
    clocks = sampler.stop() if sampler else None
    if rank != 0:
        return
    ref = next(r for r in results if r["batch"] == 1 and r["kv_len"] == 8192)
    line = {
        "metric": "measured wall-clock speedup of block decoding over NTP (k=16, NFE speedup 4, "
                  "batch 1, KV 8192)",
        "value": ref["speedup"]["k16_nfe4"], "unit": "x", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (PyTorch seeded device generator; random-init 8B-shaped weights)",
        "config": {"workload": "speedup_tables", "model": "Llama-3.1-8B shapes, 32 layers",
                   "batches": list(SPEEDUP_BATCHES), "kv_lens": list(SPEEDUP_KV_LENS),
                   "block_sizes": list(SPEEDUP_KS), "nfe_speedups": list(SPEEDUP_NFE),
                   "linear_layers": ("sbd_linear (tcgen05 LM-head kernel, storing epilogue)"
                                     if args.linear == "sbd" else "cuBLAS bf16 GEMMs (torch.matmul)"),
                   "attention_and_head": "libsbd kernels"},
        "clocks": clocks,
        "tables": results,
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="llama8b_k16",
                    choices=["llama8b_k16", "ragged_b32_k8", "qwen8b_long_k16", "tiny_f32",
                             "sweep32_k4", "sweep32_k8", "sweep32_k16", "sweep32_k32",
                             "speedup_tables"])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--gamma", type=float, default=0.1)
    ap.add_argument("--tau", type=float, default=1.0)
    ap.add_argument("--noise", choices=["buffer", "philox"], default="buffer",
                    help="Gumbel noise read from a tensor, or generated in the LM-head kernel")
    ap.add_argument("--skip-e2e", action="store_true")
    ap.add_argument("--skip-cpu", action="store_true")
    ap.add_argument("--no-graph", action="store_true", help="time eager launches, no CUDA graph")
    ap.add_argument("--linear", choices=["cublas", "sbd"], default="cublas",
                    help="GEMMs of the model's linear layers in --workload speedup_tables")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    elif args.workload.startswith("sweep32"):
        run_sweep(args)
    elif args.workload == "speedup_tables":
        run_speedup_tables(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
