#!/usr/bin/env python3
"""Benchmark of the batch-1 QTEA ternary + 1:4 residual GEMV on GB300.

Workload: the seven linear layers of one Llama3-8B decoder layer (q/k/v/o/gate/up/down, out x in
= 4096x4096, 1024x4096, 1024x4096, 4096x4096, 14336x4096, 14336x4096, 4096x14336) at batch M = 1,
with synthetic weights drawn like the paper's models would be stored (ternary codes
P(-1,0,+1) = (0.3,0.4,0.3), alpha ~ U(0.01,0.05), v ~ U(0.8,1.2), 3% salient columns, residual
~ N(0,0.02), x ~ N(0,1)). `--layers` independent layers are resident in HBM (default 32: the
whole decoder stack, 1.87 GB of codes) and the steps rotate through them, so every step reads
weights that are not in L2; `layers` consecutive steps are one token's linear layers.

A step = the seven GEMVs of one layer. value = algorithmic bytes moved per step (packed ternary
codes, alpha, v, salient indices, residual values and positions, x, y) x steps / device time.
Prints one JSON line (rank 0).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "µs/call and achieved HBM GB/s (% of GB300 peak) for batch-1 ternary+1:4 GEMV"
WORKLOAD = "llama3_8b_layer_gemvs_m1"
LAYER_WORKLOAD = "llama3_8b_layer"  # the seven GEMVs of one Llama3-8B decoder layer


def algorithmic_bytes(N, K, s, M=1):
    K_pad = -(-K // 64) * 64
    return (N * K_pad // 4 + 2 * N + 2 * K + 4 * s + 2 * (N // 4) * s + (N // 4) * ((s + 3) // 4)
            + 2 * M * K + 4 * M * N)


def paper_algorithmic_bytes(N, K, s, M=1, group=128):
    """Bytes one call must move in the paper's storage: base-3 codes (26 bytes per 128 columns),
    alpha and beta per (row, group), v, salient list, FP8 residual values, positions, x, y."""
    G = -(-K // group)
    return (N * (-(-K // 128)) * 26 + 2 * 2 * N * G + 2 * K + 4 * s + (N // 4) * s + (N // 4) * ((s + 3) // 4)
            + 2 * M * K + 4 * M * N)


def profiled_traffic():
    """DRAM bytes per launch from the committed ncu summary, if the kernel source still
    matches the one that was profiled (else None)."""
    import hashlib
    prof = os.path.join(ROOT, "profiles", "qtea_gemv_m1_llama3_8b_layer.md")
    srcs = [os.path.join(ROOT, "paper_2609_00224_gb300", "csrc", f) for f in ("qtea_gemv_m1.cu", "qtea_m1_device.h")]
    try:
        text = open(prof).read()
        sha = hashlib.sha256(b"".join(open(f, "rb").read() for f in srcs)).hexdigest()[:16]
        fields = dict(l.split(":", 1) for l in text.splitlines() if l.startswith(("kernel_source_sha256_16:",
                                                                                   "traffic_bytes_per_launch:")))
        if fields.get("kernel_source_sha256_16", "").strip() != sha:
            return None
        return int(fields["traffic_bytes_per_launch"].strip())
    except Exception:
        return None


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.thread.join(timeout=2)
        mhz, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                mhz.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not mhz:
            return None
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(mhz)}


class ExternalEvents:
    """Records a CUDA event as an event-record node while a stream is being captured
    (cuEventRecordWithFlags with CU_EVENT_RECORD_EXTERNAL), so graph replays time each launch."""

    def __init__(self):
        import ctypes
        self.ok = False
        try:
            self.cu = ctypes.CDLL("libcuda.so.1")
            self.cu.cuEventRecordWithFlags.restype = ctypes.c_int
            self.cu.cuEventRecordWithFlags.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_uint]
            self.ok = True
        except Exception:
            self.ok = False

    def record(self, event, stream):
        rc = self.cu.cuEventRecordWithFlags(event.cuda_event, stream.cuda_stream, 1)
        if rc != 0:
            raise RuntimeError(f"cuEventRecordWithFlags failed with {rc}")


# ---------------------------------------------------------------------------- workload

def make_layer(layer, torch, qt, synth, keep_host=False):
    """Generate one layer's seven problems, pack them on the device, keep device operands."""
    out = []
    for mi, (name, N, K) in enumerate(synth.workload_shapes(LAYER_WORKLOAD)):
        p = synth.workload_problem(LAYER_WORKLOAD, mi, layer=layer)
        f16 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.float16)
        T = torch.from_numpy(p.T).cuda()
        lay = qt.qtea_pack_layout(T, n_salient=p.s)
        del T
        g = dict(name=name, N=N, K=K, s=p.s, layout=lay, x=f16(p.x), alpha=f16(p.alpha.reshape(-1)), v=f16(p.v),
                 sal=torch.from_numpy(p.salient_idx).cuda(), rv=f16(p.residual_vals),
                 ri=torch.from_numpy(p.residual_idx).cuda(), y=torch.empty((1, N), dtype=torch.float32, device="cuda"),
                 bytes=algorithmic_bytes(N, K, p.s))
        if keep_host:
            g["host"] = p
        out.append(g)
    return out


def run_step(qt, layer, stream):
    for g in layer:
        qt.qtea_gemv(g["x"], g["layout"], g["alpha"], g["v"], g["sal"], g["rv"], g["ri"], y=g["y"], stream=stream)


def oracle_sample_seconds(problems, rows_stride, budget_s):
    """Time the oracle (as it stands, 1 thread) over sampled rows of the given problems."""
    import oracle
    done_bytes, t_total, n_rows_total = 0.0, 0.0, 0
    i = 0
    while t_total < budget_s and i < len(problems) * 100:
        p = problems[i % len(problems)]
        rows = np.arange(i // len(problems) % rows_stride, p.N, rows_stride, dtype=np.int32)
        t0 = time.perf_counter()
        oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx, rows=rows,
                    want_bound=False)
        t_total += time.perf_counter() - t0
        done_bytes += algorithmic_bytes(p.N, p.K, p.s) * len(rows) / p.N
        n_rows_total += len(rows)
        i += 1
    return done_bytes, t_total, n_rows_total


def _oracle_rows_worker(w, workers, stride, cmd_q, done_q):
    """One host core of the parallel oracle timing: generate the layer-0 problems once, then for
    each step compute the step's sampled rows (every stride-th row, offset by the step) that fall to
    this worker, reporting (bytes, rows, seconds)."""
    import oracle
    import synth
    probs = [synth.workload_problem(LAYER_WORKLOAD, mi, layer=0) for mi in range(7)]
    done_q.put(("ready", w))
    while True:
        cmd = cmd_q.get()
        if cmd is None:
            return
        step = cmd
        t0 = time.perf_counter()
        b, n = 0.0, 0
        for p in probs:
            rows = np.arange(step % stride, p.N, stride, dtype=np.int32)[w::workers]
            if len(rows):
                oracle.gemv(p.x, p.T, p.alpha, p.v, p.salient_idx, p.residual_vals, p.residual_idx, rows=rows,
                            want_bound=False)
            b += algorithmic_bytes(p.N, p.K, p.s) * len(rows) / p.N
            n += len(rows)
        done_q.put(("step", w, b, n, time.perf_counter() - t0))


class ParallelOracle:
    """The oracle as it stands, one process per host core (spawned, so no CUDA state is inherited),
    each taking a disjoint share of a step's sampled output rows."""

    def __init__(self, stride, workers=None):
        import multiprocessing as mp
        ctx = mp.get_context("spawn")
        self.workers = workers or len(os.sched_getaffinity(0))
        self.stride = stride
        self.done_q = ctx.Queue()
        self.cmd_qs = [ctx.Queue() for _ in range(self.workers)]
        self.procs = [ctx.Process(target=_oracle_rows_worker, args=(w, self.workers, stride, self.cmd_qs[w],
                                                                   self.done_q), daemon=True)
                      for w in range(self.workers)]
        for pr in self.procs:
            pr.start()
        for _ in range(self.workers):
            tag, _w = self.done_q.get(timeout=600)
            assert tag == "ready"

    def step(self, step):
        """One step on all workers; returns (bytes, rows, wall seconds)."""
        t0 = time.perf_counter()
        for q in self.cmd_qs:
            q.put(step)
        b, n = 0.0, 0
        for _ in range(self.workers):
            _tag, _w, bw, nw, _t = self.done_q.get(timeout=600)
            b += bw
            n += nw
        return b, n, time.perf_counter() - t0

    def close(self):
        for q in self.cmd_qs:
            q.put(None)
        for pr in self.procs:
            pr.join(timeout=60)


# ---------------------------------------------------------------------------- arms

def max_over_ranks(ms, world, device):
    """The slowest rank's time in ms (every rank receives it); ms itself on a single rank."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(bytes_per_rank, world, ms):
    """Whole-job GB/s: the bytes all ranks processed over the slowest rank's time (weak scaling)."""
    return bytes_per_rank * world / (ms * 1e-3) / 1e9


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def reference_arm(args):
    """The oracle, as it stands, on the host cores: each step a bounded sample of the workload."""
    world, rank, _ = dist_setup()
    if rank != 0:
        return 0
    import oracle
    import synth
    oracle.build()
    synth.build()
    rows_stride = 16  # every 16th output row of each of the 7 GEMVs per step
    pool = ParallelOracle(rows_stride)
    try:
        for w in range(args.warmup):
            pool.step(w)
        tot_b, tot_t, tot_rows = 0.0, 0.0, 0
        for step in range(args.steps):
            b, n, t = pool.step(step)
            tot_b += b
            tot_rows += n
            tot_t += t
    finally:
        pool.close()
    value = tot_b / tot_t / 1e9
    sample = (f"each step: every {rows_stride}th output row of the 7 Llama3-8B layer GEMVs "
              f"({tot_rows // max(args.steps, 1)} rows/step), fp64 oracle, {pool.workers} processes "
              f"(one per host core) on disjoint rows")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_t / max(args.steps, 1),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "M": 1, "note": "bounded row sample per step"},
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": pool.workers, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def qtea_arm(args):
    import torch
    import synth
    import paper_2609_00224_gb300 as qt

    world, rank, local = dist_setup()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    qt.load()
    warmup = max(args.warmup, 3)
    stream = torch.cuda.Stream()
    t_gen = time.perf_counter()
    layers = [make_layer(l, torch, qt, synth, keep_host=(l == 0 and rank == 0 and not args.no_cpu_baseline))
              for l in range(args.layers)]
    for L in layers:
        for g in L:
            g["layout"].set_activation_precision(args.act_bits)
    torch.cuda.synchronize()
    t_gen = time.perf_counter() - t_gen
    resident = sum(g["layout"].describe()["packed_bytes"] for L in layers for g in L)
    step_bytes = [sum(g["bytes"] for g in L) for L in layers]
    l2 = torch.cuda.get_device_properties(local).L2_cache_size
    launches_per_step = 7

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    # ---- CUDA graphs: the warm-up steps and the K timed steps are each captured once; the timed
    #      graph records an event before and after every launch (event-record nodes), so the
    #      per-launch durations come from the timed region itself
    ext = ExternalEvents()
    n_ev = args.steps * launches_per_step
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_ev)]
    for a_, b_ in ev:  # materialise the event handles before capture
        a_.record(stream)
        b_.record(stream)
    torch.cuda.synchronize()

    group_args = [[dict(x=g["x"], layout=g["layout"], row_scale=g["alpha"], col_scale=g["v"], salient_idx=g["sal"],
                        residual_vals=g["rv"], residual_idx=g["ri"], y=g["y"]) for g in L] for L in layers]

    def capture(steps, with_events, grouped=True, only=None):
        """One step = the 7 GEMVs of one layer as one grouped launch, or 7 single launches, or
        (only = j) GEMV j of the layer alone. Without events, consecutive launches overlap through
        programmatic dependent launch; event-record nodes between launches serialise them."""
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=stream):
            k = 0
            for st in range(steps):
                li = st % len(layers)
                if grouped:
                    if with_events:
                        ext.record(ev[k][0], stream)
                    qt.qtea_gemv_grouped(group_args[li], stream=stream)
                    if with_events:
                        ext.record(ev[k][1], stream)
                    k += 1
                    continue
                for j, gm in enumerate(layers[li]):
                    if only is not None and j != only:
                        continue
                    if with_events:
                        ext.record(ev[k][0], stream)
                    qt.qtea_gemv(gm["x"], gm["layout"], gm["alpha"], gm["v"], gm["sal"], gm["rv"], gm["ri"],
                                 y=gm["y"], stream=stream)
                    if with_events:
                        ext.record(ev[k][1], stream)
                    k += 1
        return gr

    def timed_replay(gr):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            gr.replay()  # warm replay
        barrier()
        with torch.cuda.stream(stream):
            e0.record(stream)
            gr.replay()
            e1.record(stream)
        barrier()
        return e0.elapsed_time(e1)

    g_warm = capture(warmup, False)
    g_timed = capture(args.steps, False)
    with torch.cuda.stream(stream):
        g_warm.replay()
    barrier()

    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    # the timed graph once, untimed, right before its timed replay: its first launch uploads it
    # (hundreds of kernel nodes with their parameters), which would otherwise fall between the
    # events of the timed replay, and the GPU leaves the idle of the sleep
    with torch.cuda.stream(stream):
        g_timed.replay()
    barrier()
    with torch.cuda.stream(stream):
        t_start.record(stream)
        g_timed.replay()
        t_end.record(stream)
    barrier()
    clk = clocks.stop()
    total_ms = t_start.elapsed_time(t_end)
    status = max(qt.qtea_device_status(g["layout"]) for L in layers for g in L)
    if status:
        raise RuntimeError(f"device status {status} after the timed region")
    total_ms = max_over_ranks(total_ms, world, "cuda")
    bytes_rank = sum(step_bytes[st % len(layers)] for st in range(args.steps))
    bytes_all = bytes_rank * world
    value = job_throughput(bytes_rank, world, total_ms)

    # roofline of the GEMV kernel: the only kernel of the timed region, one grouped launch per
    # step, launches back to back; its average launch duration is the region time / launches
    kern_bytes = sum(step_bytes[st % len(layers)] for st in range(args.steps))
    achieved = kern_bytes / (total_ms * 1e-3) / 1e9
    peak, peak_src = load_peaks()
    # the same launches one at a time (event-record nodes between them), for the isolated duration
    iso_us = None
    if ext.ok:
        g_ev = capture(args.steps, True)
        timed_replay(g_ev)
        iso_us = statistics.mean(a_.elapsed_time(b_) for a_, b_ in ev[:args.steps]) * 1e3
        del g_ev

    # ---- per-GEMV latency: each GEMV of the layer alone, launched back to back over the layers
    per_shape = {}
    if not args.no_per_shape:
        for j, gm in enumerate(layers[0]):
            gs = capture(args.steps, False, grouped=False, only=j)
            ms = timed_replay(gs)
            del gs
            us = ms * 1e3 / args.steps
            N, K = gm["N"], gm["K"]
            bts = statistics.mean(L[j]["bytes"] for L in layers)
            per_shape[gm["name"]] = {"N": N, "K": K, "s": gm["s"], "us_per_call": round(us, 3),
                                     "kernel": qt.qtea_gemv_plan([group_args[0][j]])[0],
                                     "gbs": round(bts / (us * 1e-6) / 1e9, 1),
                                     "eff_bits_per_weight": round(8 * (bts - 2 * K - 4 * N) / (N * K), 3)}

    # ---- the 32-layer stack in a decoder's dependency order: per layer four grouped calls
    #      (q, k, v | o | gate, up | down), every layer of the stack once per token, the tokens
    #      back to back in one graph (x per GEMV synthetic, not chained)
    stack = None
    if not args.no_stack and len(layers) >= 2:
        order = [[0, 1, 2], [3], [4, 5], [6]]
        n_tok = max(2, min(8, args.steps // len(layers)))
        gs_ = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            for L in group_args:
                for grp in order:
                    qt.qtea_gemv_grouped([L[j] for j in grp], stream=stream)
        barrier()
        with torch.cuda.graph(gs_, stream=stream):
            for _ in range(n_tok):
                for L in group_args:
                    for grp in order:
                        qt.qtea_gemv_grouped([L[j] for j in grp], stream=stream)
        ms_s = timed_replay(gs_)
        del gs_
        tok_b = sum(step_bytes)
        kern = {name: qt.qtea_gemv_plan([group_args[0][j] for j in grp])[0]
                for name, grp in zip(("q_k_v", "o", "gate_up", "down"), order)}
        stack = {"workload": f"llama3_8b_stack_{len(layers)}_layers_dependency_order", "tokens": n_tok,
                 "launches_per_token": 4 * len(layers), "kernels": kern, "us_per_token": round(ms_s * 1e3 / n_tok, 1),
                 "linear_tokens_per_s": round(n_tok / (ms_s * 1e-3), 1),
                 "GBps": round(tok_b * n_tok / (ms_s * 1e-3) / 1e9, 1),
                 "frac_of_measured_hbm": round(tok_b * n_tok / (ms_s * 1e-3) / 1e9 / peak, 3)}

    # ---- the other activation precision, same steps (reported beside the headline mode)
    alt = {}
    other = 16 if args.act_bits == 24 else 24
    for L in layers:
        for g in L:
            g["layout"].set_activation_precision(other)
    g_alt = capture(args.steps, False)
    with torch.cuda.stream(stream):
        g_alt.replay()
    barrier()
    ea, eb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        ea.record(stream)
        g_alt.replay()
        eb.record(stream)
    barrier()
    alt_ms = ea.elapsed_time(eb)
    alt[f"act{other}"] = {"value": round(kern_bytes / (alt_ms * 1e-3) / 1e9, 1), "unit": "GB/s",
                          "ms_per_step": round(alt_ms / args.steps, 5)}
    for L in layers:
        for g in L:
            g["layout"].set_activation_precision(args.act_bits)
    del g_alt

    # ---- end to end through the public API with host buffers (pinned), copies inside the region: per
    #      step the seven x vectors go to the device in one copy (a contiguous pinned staging buffer
    #      holds them, as a caller would lay them out), the grouped call runs on views of one device
    #      buffer, and the seven y vectors come back in one copy
    e2e = None
    if not args.no_e2e:
        L0 = layers
        ks = [g["K"] for g in L0[0]]
        ns = [g["N"] for g in L0[0]]
        xo = np.concatenate([[0], np.cumsum(ks)]).tolist()
        yo = np.concatenate([[0], np.cumsum(ns)]).tolist()
        # pinned inputs per layer; per step its own device input, device output and pinned output
        n_buf = max(args.steps, warmup)
        hx = [torch.cat([g["x"].reshape(-1).cpu() for g in L]).pin_memory() for L in L0]
        hy = [torch.empty(yo[-1], dtype=torch.float32).pin_memory() for _ in range(n_buf)]
        dx = [torch.empty(xo[-1], dtype=torch.float16, device="cuda") for _ in range(n_buf)]
        dy = [torch.empty(yo[-1], dtype=torch.float32, device="cuda") for _ in range(n_buf)]
        eargs = [[dict(x=dx[b][xo[j]:xo[j + 1]].view(1, ks[j]), layout=g["layout"], row_scale=g["alpha"],
                       col_scale=g["v"], salient_idx=g["sal"], residual_vals=g["rv"], residual_idx=g["ri"],
                       y=dy[b][yo[j]:yo[j + 1]].view(1, ns[j])) for j, g in enumerate(L0[b % len(L0)])]
                 for b in range(n_buf)]
        h2d = 2 * xo[-1]
        d2h = 4 * yo[-1]

        # Each step: its inputs copied in (one copy on a copy stream, issued with those of the next
        # seven steps), its grouped call (compute stream, after its batch of copies), its results
        # copied out (one copy on an output stream, after the call). Every step has its own buffers,
        # so the copies overlap the grouped calls; only the first call of each batch of eight waits
        # on a copy, and the other calls follow each other with programmatic dependent launch.
        s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
        e2e_batch = 8

        def e2e_steps(n):
            s_in.wait_stream(stream)
            s_out.wait_stream(stream)
            for st in range(n):
                if st % e2e_batch == 0:
                    with torch.cuda.stream(s_in):
                        for b in range(st, min(n, st + e2e_batch)):
                            dx[b].copy_(hx[b % len(L0)], non_blocking=True)
                        ev_in = torch.cuda.Event()
                        ev_in.record(s_in)
                    stream.wait_event(ev_in)
                with torch.cuda.stream(stream):
                    qt.qtea_gemv_grouped(eargs[st], stream=stream)
                    ev_k = torch.cuda.Event()
                    ev_k.record(stream)
                s_out.wait_event(ev_k)
                with torch.cuda.stream(s_out):
                    hy[st].copy_(dy[st], non_blocking=True)
            stream.wait_stream(s_in)
            stream.wait_stream(s_out)

        with torch.cuda.stream(stream):
            e2e_steps(warmup)
        barrier()
        ge = torch.cuda.CUDAGraph()
        with torch.cuda.graph(ge, stream=stream):
            e2e_steps(args.steps)
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            ge.replay()
            e1.record(stream)
        barrier()
        e2e_ms = e0.elapsed_time(e1)
        e2e_ms = max_over_ranks(e2e_ms, world, "cuda")
        e2e = {"value": round(job_throughput(bytes_rank, world, e2e_ms), 1), "unit": "GB/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": round(e2e_ms / args.steps, 5),
               "copies_per_step": {"h2d": 1, "d2h": 1},
               "overlap": "input copies issued eight steps at a time on a copy stream, output copies on a "
                          "third stream after each call; copies overlap the grouped calls"}

    # ---- dense fp16 GEMV through cuBLAS (torch.mm) on the same seven shapes: the
    #      unquantized baseline, weights in enough copies that every step reads them from HBM
    dense = None
    if not args.no_dense:
        copies = max(2, -(-4 * l2 // sum(2 * g["N"] * g["K"] for g in layers[0])))
        dw = [[torch.randn((g["N"], g["K"]), dtype=torch.float16, device="cuda") for g in layers[0]]
              for _ in range(copies)]
        dx = [torch.randn((1, g["K"]), dtype=torch.float16, device="cuda") for g in layers[0]]
        dy = [torch.empty((1, g["N"]), dtype=torch.float16, device="cuda") for g in layers[0]]

        with torch.cuda.stream(stream):  # cuBLAS creates its handle and workspace outside the capture
            for j in range(len(dx)):
                torch.mm(dx[j], dw[0][j].t(), out=dy[j])
        barrier()

        def dense_graph(only=None):
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=stream):
                for st in range(args.steps):
                    for j in range(len(dx)):
                        if only is None or j == only:
                            torch.mm(dx[j], dw[st % copies][j].t(), out=dy[j])
            return gr

        gd = dense_graph()
        dms = timed_replay(gd)
        del gd
        dbytes = sum(2 * g["N"] * g["K"] + 2 * g["K"] + 2 * g["N"] for g in layers[0])
        dense = {"us_per_step": round(dms * 1e3 / args.steps, 3), "value": round(dbytes * args.steps / (dms * 1e-3) / 1e9, 1),
                 "unit": "GB/s", "weight_copies": copies, "us_per_call": {}}
        if not args.no_per_shape:
            for j, g in enumerate(layers[0]):
                gs = dense_graph(only=j)
                dense["us_per_call"][g["name"]] = round(timed_replay(gs) * 1e3 / args.steps, 3)
                del gs
        dense["qtea_speedup_per_step"] = round(dense["us_per_step"] / (1e3 * total_ms / args.steps), 2)
        del dw, dx, dy
        torch.cuda.empty_cache()

    # ---- Qwen3-14B layer shapes at batch M = 1 .. 16 (reported beside the batch-1 workload): the seven
    #      GEMVs of a layer per step, rotating over resident layers; the dense fp16 GEMM on the same shapes
    msweep = None
    if not args.no_m_sweep:
        msweep = {"workload": "qwen3_14b_layer_gemvs", "layers_resident": 4, "us_per_layer": {}}
        qlayers = []
        for li in range(4):
            L = []
            for mi, (name, N, K) in enumerate(synth.workload_shapes("qwen3_14b_layer")):
                pq = synth.workload_problem("qwen3_14b_layer", mi, M=16, layer=li)
                f16 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.float16)
                T = torch.from_numpy(pq.T).cuda()
                lay = qt.qtea_pack_layout(T, n_salient=pq.s)
                del T
                L.append(dict(layout=lay, x=f16(pq.x), alpha=f16(pq.alpha.reshape(-1)), v=f16(pq.v),
                              sal=torch.from_numpy(pq.salient_idx).cuda(), rv=f16(pq.residual_vals),
                              ri=torch.from_numpy(pq.residual_idx).cuda(), N=N, K=K))
            qlayers.append(L)
        qcopies = 2
        qw = [[torch.randn((g["N"], g["K"]), dtype=torch.float16, device="cuda") for g in qlayers[0]]
              for _ in range(qcopies)]
        nsteps = 32
        for M in (1, 2, 4, 8, 16):
            ys = [[torch.empty((M, g["N"]), dtype=torch.float32, device="cuda") for g in L] for L in qlayers]
            yd = [torch.empty((M, g["N"]), dtype=torch.float16, device="cuda") for g in qlayers[0]]
            xs = [[g["x"][:M].contiguous() for g in L] for L in qlayers]

            def qstep(st):
                L = qlayers[st % len(qlayers)]
                qt.qtea_gemv_grouped([dict(x=xs[st % len(qlayers)][j], layout=g["layout"], row_scale=g["alpha"],
                                           col_scale=g["v"], salient_idx=g["sal"], residual_vals=g["rv"],
                                           residual_idx=g["ri"], y=ys[st % len(qlayers)][j])
                                      for j, g in enumerate(L)], stream=stream)

            def dstep(st):
                for j in range(len(yd)):
                    torch.mm(xs[0][j], qw[st % qcopies][j].t(), out=yd[j])

            with torch.cuda.stream(stream):
                qstep(0)
                dstep(0)
            barrier()
            gq = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gq, stream=stream):
                for st in range(nsteps):
                    qstep(st)
            tq = timed_replay(gq) * 1e3 / nsteps
            gdd = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gdd, stream=stream):
                for st in range(nsteps):
                    dstep(st)
            tdn = timed_replay(gdd) * 1e3 / nsteps
            del gq, gdd
            lb = sum(algorithmic_bytes(g["N"], g["K"], g["sal"].numel(), M) for g in qlayers[0])
            msweep["us_per_layer"][str(M)] = {"qtea": round(tq, 2), "dense_fp16": round(tdn, 2),
                                              "speedup": round(tdn / tq, 2), "GBps": round(lb / tq / 1e3, 1),
                                              "frac_of_measured_hbm": round(lb / tq / 1e3 / peak, 3)}
        status = max(qt.qtea_device_status(g["layout"]) for L in qlayers for g in L)
        if status:
            raise RuntimeError(f"device status {status} after the batch sweep")
        del qlayers, qw
        torch.cuda.empty_cache()

    # ---- the Llama3-8B layer in the paper's own storage (base-3 codes, alpha and beta per 128-column
    #      group, FP8 residual values), and with the paper's scale groups on 2-bit codes and fp16
    #      residual values: the seven GEMVs per step as one grouped call, rotating over resident layers
    def paper_leg(fmt, fp8):
        n_res = 4
        players = []
        for li in range(n_res):
            L = []
            for mi in range(7):
                pp = synth.paper_problem("llama3_8b_layer", mi, layer=li, residual_fp8=fp8)
                f16 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.float16)
                T = torch.from_numpy(pp.T).cuda()
                lay = qt.qtea_pack_layout(T, n_salient=pp.s, group_size=128, fmt=fmt)
                lay.set_options(qt.QTEA_OPT_BIAS | (qt.QTEA_OPT_RESIDUAL_FP8 if fp8 else 0))
                del T
                sc = np.stack([pp.alpha.reshape(pp.N, -1), pp.beta.reshape(pp.N, -1)], axis=-1).reshape(-1)
                rv = torch.from_numpy(pp.residual_vals).cuda() if fp8 else f16(pp.residual_vals)
                L.append(dict(x=f16(pp.x), layout=lay, row_scale=f16(sc), col_scale=f16(pp.v),
                              salient_idx=torch.from_numpy(pp.salient_idx).cuda(), residual_vals=rv,
                              residual_idx=torch.from_numpy(pp.residual_idx).cuda(),
                              y=torch.empty((1, pp.N), dtype=torch.float32, device="cuda")))
            players.append(L)
        shapes = synth.workload_shapes("llama3_8b_layer")
        if fmt == qt.QTEA_FMT_BASE3 and fp8:
            pbytes = sum(paper_algorithmic_bytes(N, K, synth.salient_count(K)) for _, N, K in shapes)
        else:
            # 2-bit codes and fp16 residual values with (alpha, beta) per 128-column group
            pbytes = sum(algorithmic_bytes(N, K, synth.salient_count(K)) + 4 * N * (-(-K // 128)) - 2 * N
                         for _, N, K in shapes)
        nsteps = 16
        with torch.cuda.stream(stream):
            qt.qtea_gemv_grouped(players[0], stream=stream)
        gp = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gp, stream=stream):
            for st in range(nsteps):
                qt.qtea_gemv_grouped(players[st % n_res], stream=stream)
        tp = timed_replay(gp) * 1e3 / nsteps
        del gp
        status = max(qt.qtea_device_status(g["layout"]) for L in players for g in L)
        if status:
            raise RuntimeError(f"device status {status} in the paper-storage steps")
        w = sum(N * K for _, N, K in shapes)
        res = {"us_per_step": round(tp, 2), "GBps": round(pbytes / (tp * 1e-6) / 1e9, 1),
               "frac_of_measured_hbm": round(pbytes / (tp * 1e-6) / 1e9 / peak, 3), "bytes_per_step": pbytes,
               "bits_per_weight": round(8 * (pbytes - sum(2 * K + 4 * N for _, N, K in shapes)) / w, 3),
               "layers_resident": n_res}
        del players
        torch.cuda.empty_cache()
        return res

    paper = None
    if not args.no_paper:
        paper = {"workload": "llama3_8b_layer_paper_storage", "M": 1,
                 "base3_fp8": dict(paper_leg(qt.QTEA_FMT_BASE3, True),
                                   kernel="qtea_gemv_lut_kernel<grouped> (the paper's table decode, alpha and "
                                          "beta per 128 columns staged per tile)"),
                 "2bit_fp16_residual": dict(paper_leg(qt.QTEA_FMT_2BIT, False),
                                            kernel="qtea_gemv_m1_kernel, grouped variant (alpha and beta "
                                                   "applied per 128-column group in the decode)")}

    # ---- the paper's decode against the fixed-point one: the Llama3-8B layer in base-3 codes (one
    #      alpha per row, fp16 residual values), the same resident layouts decoded by the sign-symmetric
    #      lookup table (Sec. 3.5, Appendix A) and by the fixed-point dot-product kernel
    def lut_leg():
        n_res, nsteps = 4, 16
        shapes = synth.workload_shapes(LAYER_WORKLOAD)
        players = []
        for li in range(n_res):
            L = []
            for mi in range(7):
                pp = synth.workload_problem(LAYER_WORKLOAD, mi, layer=li)
                f16 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.float16)
                T = torch.from_numpy(pp.T).cuda()
                lay = qt.qtea_pack_layout(T, n_salient=pp.s, fmt=qt.QTEA_FMT_BASE3)
                del T
                L.append(dict(x=f16(pp.x), layout=lay, row_scale=f16(pp.alpha.reshape(-1)), col_scale=f16(pp.v),
                              salient_idx=torch.from_numpy(pp.salient_idx).cuda(), residual_vals=f16(pp.residual_vals),
                              residual_idx=torch.from_numpy(pp.residual_idx).cuda(),
                              y=torch.empty((1, pp.N), dtype=torch.float32, device="cuda")))
            players.append(L)
        # base-3 codes, one alpha per row, fp16 residual values
        pbytes = sum(algorithmic_bytes(N, K, synth.salient_count(K)) - N * (-(-K // 64) * 64) // 4
                     + N * (-(-K // 128)) * 26 for _, N, K in shapes)
        out = {}
        for name, opt in (("lut", 0), ("fixed_point_dp4a", qt.QTEA_OPT_FIXED_POINT)):
            for L in players:
                for g in L:
                    g["layout"].set_options(opt)
            with torch.cuda.stream(stream):
                qt.qtea_gemv_grouped(players[0], stream=stream)
            gp = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gp, stream=stream):
                for st in range(nsteps):
                    qt.qtea_gemv_grouped(players[st % n_res], stream=stream)
            tp = timed_replay(gp) * 1e3 / nsteps
            del gp
            status = max(qt.qtea_device_status(g["layout"]) for L in players for g in L)
            if status:
                raise RuntimeError(f"device status {status} in the {name} steps")
            out[name] = {"us_per_step": round(tp, 2), "GBps": round(pbytes / (tp * 1e-6) / 1e9, 1),
                         "frac_of_measured_hbm": round(pbytes / (tp * 1e-6) / 1e9 / peak, 3)}
        out["lut"]["kernel"] = "qtea_gemv_lut_kernel (half-LUT of 122 fp32 entries per code byte)"
        out["fixed_point_dp4a"]["kernel"] = "qtea_gemv_paper_b3_kernel (22/23-bit planes, dp4a)"
        out["bytes_per_step"] = pbytes
        out["layers_resident"] = n_res
        del players
        torch.cuda.empty_cache()
        return out

    lut = None
    if not args.no_paper:
        lut = {"workload": "llama3_8b_layer_base3_one_alpha_per_row", "M": 1, **lut_leg()}

    # ---- the Llama3-70B layer (8192-wide, 28672-row MLP: the large-K shapes) at M = 1, the seven
    #      GEMVs per step as one grouped call, rotating over resident layers whose codes exceed L2
    def llama70b_leg():
        wl, n_res, nsteps = "llama3_70b_layer", 3, 24
        shapes = synth.workload_shapes(wl)
        players, pbytes = [], []
        for li in range(n_res):
            L, b = [], 0
            for mi, (_, N, K) in enumerate(shapes):
                pp = synth.workload_problem(wl, mi, layer=li)
                f16 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.float16)
                T = torch.from_numpy(pp.T).cuda()
                lay = qt.qtea_pack_layout(T, n_salient=pp.s)
                lay.set_activation_precision(args.act_bits)
                del T
                L.append(dict(x=f16(pp.x), layout=lay, row_scale=f16(pp.alpha.reshape(-1)), col_scale=f16(pp.v),
                              salient_idx=torch.from_numpy(pp.salient_idx).cuda(), residual_vals=f16(pp.residual_vals),
                              residual_idx=torch.from_numpy(pp.residual_idx).cuda(),
                              y=torch.empty((1, N), dtype=torch.float32, device="cuda")))
                b += algorithmic_bytes(N, K, pp.s)
            players.append(L)
            pbytes.append(b)
        codes = sum(g["layout"].describe()["packed_bytes"] for L in players for g in L)
        with torch.cuda.stream(stream):
            qt.qtea_gemv_grouped(players[0], stream=stream)
        gp = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gp, stream=stream):
            for st in range(nsteps):
                qt.qtea_gemv_grouped(players[st % n_res], stream=stream)
        ms = timed_replay(gp)
        del gp
        status = max(qt.qtea_device_status(g["layout"]) for L in players for g in L)
        if status:
            raise RuntimeError(f"device status {status} in the Llama3-70B steps")
        tb = sum(pbytes[st % n_res] for st in range(nsteps))
        gbs = tb / (ms * 1e-3) / 1e9
        res = {"workload": "llama3_70b_layer_gemvs", "M": 1, "us_per_step": round(ms * 1e3 / nsteps, 2),
               "GBps": round(gbs, 1), "frac_of_measured_hbm": round(gbs / peak, 3),
               "bytes_per_step": round(tb / nsteps), "layers_resident": n_res, "resident_code_bytes": codes,
               "act_bits": args.act_bits, "kernel": "qtea_gemv_m1_kernel (one grouped launch per step)"}
        del players
        torch.cuda.empty_cache()
        return res

    l70 = None
    if not args.no_70b:
        l70 = llama70b_leg()

    # ---- the quantizer's per-layer steps (scores, top-s, group fit, column rescale, binary16 scales,
    #      1:4 residual) on the Llama3-8B layer's seven fp32 weight matrices: 128-column groups with
    #      beta, 4 alpha refits, 2 rescale rounds, the GEMV's salient count
    def quant_leg():
        shapes = synth.workload_shapes("llama3_8b_layer")
        gen = torch.Generator(device="cuda").manual_seed(1234)
        mats = []
        for _, N, K in shapes:
            W = (torch.randn(N, K, device="cuda", generator=gen) * 0.02).half().float()
            h = torch.exp(torch.randn(K, device="cuda", generator=gen)).half().float()
            mats.append((W, h, synth.salient_count(K)))
        stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(stream):
            for W, h, s in mats:  # warm-up (allocator pool, caches)
                qt.qtea_quantize(W, h, group_size=128, n_salient=s, bias=True, stream=stream)
        stream.synchronize()
        reps = 3
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        with torch.cuda.stream(stream):
            for _ in range(reps):
                for W, h, s in mats:
                    qt.qtea_quantize(W, h, group_size=128, n_salient=s, bias=True, stream=stream)
        e1.record(stream)
        stream.synchronize()
        ms = e0.elapsed_time(e1) / reps
        w = sum(N * K for _, N, K in shapes)
        del mats
        torch.cuda.empty_cache()
        return {"workload": "llama3_8b_layer_fp32_weights", "ms_per_layer": round(ms, 3),
                "Mweights_per_s": round(w / (ms * 1e-3) / 1e6, 1),
                "W_read_GBps_once": round(4 * w / (ms * 1e-3) / 1e9, 1),
                "settings": {"group": 128, "bias": True, "fit_iters": 4, "rescale_iters": 2},
                "bit_identical_to": "oracle/quantize.py (tests/test_gpu_quantize.py)"}

    quant = None
    if not args.no_quant:
        quant = quant_leg()

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        probs = [g["host"] for g in layers[0]]
        b, t, rows = oracle_sample_seconds(probs, 16, args.cpu_seconds)
        cpu = {"value": round(b / t / 1e9, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": f"{rows} output rows (every 16th row, cycling over the 7 layer-0 GEMVs) for "
                         f"{t:.1f} s, fp64, 1 thread"}
        if not args.no_cpu_all_cores:
            pool = ParallelOracle(16)
            try:
                pb, pn, pt, st = 0.0, 0, 0.0, 0
                while pt < args.cpu_seconds:
                    b_, n_, t_ = pool.step(st)
                    pb, pn, pt, st = pb + b_, pn + n_, pt + t_, st + 1
            finally:
                pool.close()
            cpu["all_cores"] = {"value": round(pb / pt / 1e9, 4), "unit": "GB/s", "cores": pool.workers,
                                "kind": "oracle",
                                "sample": f"{pn} output rows ({st} steps of every 16th row of the 7 layer-0 "
                                          f"GEMVs) in {pt:.1f} s, fp64, one process per core on disjoint rows"}

    traffic = profiled_traffic()

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": "GB/s", "n_gpus": world, "steps": args.steps,
            "warmup": warmup, "ms_per_step": round(total_ms / args.steps, 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None,
            "dtype": f"i32 dp4a (2-bit codes x {args.act_bits}-bit fixed-point v*x) + fp32",
            "data": "synthetic",
            "config": {"workload": WORKLOAD, "M": 1, "shapes": [[g["name"], g["N"], g["K"], g["s"]] for g in layers[0]],
                       "layers_resident": args.layers, "resident_weight_bytes": resident, "l2_bytes": l2,
                       "l2": "inputs larger than L2: steps rotate over the resident layers",
                       "parallelism": "replicas" if world > 1 else "single"},
            "us_per_call": per_shape,
            # the 32-layer decode stack, called in a decoder's dependency order (4 calls per layer)
            "linear_tokens_per_s": None if stack is None else stack["linear_tokens_per_s"],
            "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                         "frac": round(achieved / peak, 4), "peak_source": peak_src, "traffic": traffic,
                         "kernel": "qtea_gemv_m1_kernel", "launches_timed": args.steps,
                         "us_per_launch": round(1e3 * total_ms / args.steps, 3),
                         "us_per_launch_isolated": None if iso_us is None else round(iso_us, 3)},
            "cpu_baseline": cpu, "dense_fp16_cublas": dense, "batch_sweep": msweep, "paper_storage": paper, "lut_vs_fixed_point": lut, "decode_stack": stack, "llama3_70b_layer": l70, "quantizer": quant, "e2e": e2e, "clocks": clk, "act_bits": args.act_bits, "other_precision": alt, "gpu_launches": args.steps, "launch": "one grouped launch per step (7 GEMVs)", "graphs": True,
            "timed_graph_replayed_untimed_first": True,
            "setup_s": round(t_gen, 1),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def profile_case(args):
    """Small fixed workloads for ncu captures, one per kernel path; each runs `--calls` calls over
    `--profile-layers` resident layers (their codes exceed L2 with the default 4), then checks the
    device status. Prints one line; times nothing.

      qwen3_14b_layer        the Qwen3-14B layer's seven GEMVs at batch --m, grouped (low-batch
                             kernel; batch-1 kernel at --m 1)
      llama3_8b_layer        the Llama3-8B layer's seven GEMVs at batch 1, grouped (batch-1 stream-K
                             kernel)
      llama3_8b_qkv          the layer's q, k and v at batch 1, grouped (row-resident batch-1 kernel,
                             two CTAs per SM), then o alone (one CTA per SM)
      llama3_8b_base3        the same in base-3 codes, one alpha per row (table-lookup kernel;
                             --fixed-point: the fixed-point base-3 kernel)
      llama3_8b_paper        the paper's storage (base-3, alpha and beta per 128 columns, FP8
                             residual) at batch --m (fixed-point base-3 kernel for --m <= 4, the
                             general paper kernel above)
      llama3_8b_paper_2bit   2-bit codes with one (alpha, beta) per row and FP8 residual values at
                             batch --m (staged paper kernel for --m <= 4)
      unaligned_residual     Qwen3-14B q_proj at batch --m with residual arrays off 16-byte
                             boundaries (low-batch prep kernel, then the main kernel)
      pack                   packing of the Llama3-8B layer's codes, 2-bit and base-3
      quantize               the quantizer on the Llama3-8B layer's seven weight matrices
    """
    import numpy as np
    import torch
    import paper_2609_00224_gb300 as qt
    import synth
    qt.load()
    case, M, n_layers = args.profile_case, args.m, args.profile_layers

    def f16(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.float16)

    def layer(wl, li, make, fmt=qt.QTEA_FMT_2BIT, group=None, opts=0, M_=1):
        out = []
        for mi in range(7):
            p = make(wl, mi, li, M_)
            lay = qt.qtea_pack_layout(torch.from_numpy(p.T).cuda(), n_salient=p.s, group_size=group or p.K, fmt=fmt)
            lay.set_options(opts)
            if p.beta is not None:
                sc = np.stack([p.alpha.reshape(p.N, -1), p.beta.reshape(p.N, -1)], axis=-1).reshape(-1)
            else:
                sc = p.alpha.reshape(-1)
            rv = torch.from_numpy(p.residual_vals).cuda() if p.residual_fp8 else f16(p.residual_vals)
            out.append(dict(x=f16(p.x), layout=lay, row_scale=f16(sc), col_scale=f16(p.v),
                            salient_idx=torch.from_numpy(p.salient_idx).cuda(), residual_vals=rv,
                            residual_idx=torch.from_numpy(p.residual_idx).cuda(),
                            y=torch.empty((M_, p.N), dtype=torch.float32, device="cuda")))
        return out

    work = lambda wl, mi, li, M_: synth.workload_problem(wl, mi, M=M_, layer=li)
    layers = []
    if case == "qwen3_14b_layer":
        layers = [layer("qwen3_14b_layer", li, work, M_=M) for li in range(n_layers)]
    elif case == "llama3_8b_layer":
        layers = [layer("llama3_8b_layer", li, work) for li in range(n_layers)]
    elif case == "llama3_8b_qkv":
        full = [layer("llama3_8b_layer", li, work) for li in range(n_layers)]
        layers = [g for L in full for g in (L[:3], L[3:4])]
    elif case == "llama3_8b_base3":
        opts = qt.QTEA_OPT_FIXED_POINT if args.fixed_point else 0
        layers = [layer("llama3_8b_layer", li, work, fmt=qt.QTEA_FMT_BASE3, opts=opts) for li in range(n_layers)]
    elif case == "llama3_8b_paper":
        paper = lambda wl, mi, li, M_: synth.paper_problem(wl, mi, M=M_, layer=li)
        layers = [layer("llama3_8b_layer", li, paper, fmt=qt.QTEA_FMT_BASE3, group=128,
                        opts=qt.QTEA_OPT_BIAS | qt.QTEA_OPT_RESIDUAL_FP8, M_=M) for li in range(n_layers)]
    elif case == "llama3_8b_paper_2bit":
        bias_row = lambda wl, mi, li, M_: synth.make_problem(
            "bias", *synth.workload_shapes(wl)[mi][1:], M_, synth.salient_count(synth.workload_shapes(wl)[mi][2]),
            synth.workload_seed(wl, li, mi), beta_std=0.002, residual_fp8=True)
        layers = [layer("llama3_8b_layer", li, bias_row, opts=qt.QTEA_OPT_BIAS | qt.QTEA_OPT_RESIDUAL_FP8, M_=M)
                  for li in range(n_layers)]
    elif case == "unaligned_residual":
        for li in range(n_layers):
            p = synth.workload_problem("qwen3_14b_layer", 0, M=M, layer=li)
            lay = qt.qtea_pack_layout(torch.from_numpy(p.T).cuda(), n_salient=p.s)
            rvb = torch.zeros(p.residual_vals.size + 1, dtype=torch.float16, device="cuda")
            rvb[1:] = f16(p.residual_vals).reshape(-1)
            layers.append([dict(x=f16(p.x), layout=lay, row_scale=f16(p.alpha.reshape(-1)), col_scale=f16(p.v),
                                salient_idx=torch.from_numpy(p.salient_idx).cuda(),
                                residual_vals=rvb[1:].view(p.residual_vals.shape),
                                residual_idx=torch.from_numpy(p.residual_idx).cuda(),
                                y=torch.empty((M, p.N), dtype=torch.float32, device="cuda"))])
    elif case == "pack":
        for li in range(args.calls):
            for mi in range(7):
                p = synth.workload_problem("llama3_8b_layer", mi, layer=li)
                T = torch.from_numpy(p.T).cuda()
                for fmt in (qt.QTEA_FMT_2BIT, qt.QTEA_FMT_BASE3):
                    qt.qtea_pack_layout(T, n_salient=p.s, fmt=fmt)
        torch.cuda.synchronize()
        print(json.dumps({"profile_case": case, "calls": args.calls, "status": 0}))
        return 0
    elif case == "quantize":
        mats = []
        for mi, (_, N, K) in enumerate(synth.workload_shapes("llama3_8b_layer")):
            W, h = synth.quant_problem(1000 + mi, N, K)
            mats.append((torch.from_numpy(W).cuda(), torch.from_numpy(h).cuda(), synth.salient_count(K)))
        for _ in range(args.calls):
            for W, h, s_ in mats:
                qt.qtea_quantize(W, h, group_size=128, n_salient=s_, bias=True)
        torch.cuda.synchronize()
        print(json.dumps({"profile_case": case, "calls": args.calls, "status": 0}))
        return 0
    for c in range(args.calls):
        qt.qtea_gemv_grouped(layers[c % len(layers)])
    torch.cuda.synchronize()
    status = max(qt.qtea_device_status(g["layout"]) for L in layers for g in L)
    print(json.dumps({"profile_case": case, "M": M, "calls": args.calls, "status": status}))
    return 1 if status else 0


def probe_decode():
    """Issue rates behind the batch-1 decode choice: cycles per instruction per SM sub-partition of
    mma.sync with constant operands and with A built from a changing word (as a decode builds it), and
    of dp4a; weights per clock per SM at batch 1 follow from the useful products per instruction."""
    import torch
    import paper_2609_00224_gb300 as qt
    torch.cuda.set_device(0)
    r = qt.qtea_probe_decode_rates()
    useful = {"mma_m16n8k16_f16_constant": 256, "mma_m16n8k16_f16_decoded_a": 256, "mma_m16n8k32_e4m3_constant": 512,
              "mma_m16n8k32_e4m3_decoded_a": 512,
              "dp4a": 64}  # weights per warp instruction at batch 1 (dp4a: 32 lanes x 4 bytes, 2 planes at 16 bits)
    per_sm = {k: round(4 * useful[k] / v, 1) for k, v in r.items()}
    print(json.dumps({"probe": "decode_issue_rates", "cycles_per_instruction_per_smsp": r,
                      "batch1_weights_per_clock_per_sm_bound": per_sm,
                      "note": "one instruction stream per chain; the decode adds its own mask and load instructions"}))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["qtea", "reference"], default="qtea")
    ap.add_argument("--no-dense", action="store_true", help="skip the dense fp16 cuBLAS baseline")
    ap.add_argument("--no-m-sweep", action="store_true", help="skip the Qwen3-14B batch sweep (M = 1 .. 16)")
    ap.add_argument("--no-paper", action="store_true", help="skip the layer in the paper's own storage")
    ap.add_argument("--no-quant", action="store_true", help="skip the quantizer timing")
    ap.add_argument("--no-70b", action="store_true", help="skip the Llama3-70B layer steps")
    ap.add_argument("--no-stack", action="store_true", help="skip the stack in dependency order")
    ap.add_argument("--layers", type=int, default=32,
                    help="independent resident layers the steps rotate over (32 = the whole Llama3-8B stack)")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-cpu-all-cores", action="store_true", help="skip the oracle timing on all host cores")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-per-shape", action="store_true")
    ap.add_argument("--act-bits", type=int, choices=[16, 24], default=16,
                    help="activation precision of the timed region (24 = exact default, 16 = fast mode)")
    ap.add_argument("--profile-case", choices=["qwen3_14b_layer", "llama3_8b_layer", "llama3_8b_qkv", "llama3_8b_base3",
                                               "llama3_8b_paper", "llama3_8b_paper_2bit", "unaligned_residual",
                                               "pack", "quantize"], default=None,
                    help="run a small fixed workload for profilers instead of the benchmark")
    ap.add_argument("--m", type=int, default=2, help="batch of --profile-case")
    ap.add_argument("--profile-layers", type=int, default=4, help="resident layers of --profile-case")
    ap.add_argument("--fixed-point", action="store_true", help="--profile-case llama3_8b_base3: fixed-point kernel")
    ap.add_argument("--calls", type=int, default=3, help="grouped calls of --profile-case")
    ap.add_argument("--probe-decode", action="store_true",
                    help="print the issue rates behind the batch-1 decode choice (dp4a against mma.sync) and exit")
    args = ap.parse_args()
    if args.profile_case:
        return profile_case(args)
    if args.probe_decode:
        return probe_decode()
    if args.impl == "reference":
        return reference_arm(args)
    return qtea_arm(args)


if __name__ == "__main__":
    sys.exit(main())
