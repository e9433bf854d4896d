"""Benchmark of query-time evidence retrieval on the 1-hour shallow index.

Workload (one stream per GPU): 4 shallow layers, 28 query / 4 key heads, d = 128,
3600 frames x 196 visual tokens (705,600 keys per (layer, key head), 2.89 GB of bf16
keys), keys ~N(0,1) with 2 outlier channels x8 and per-frame AR(1) drift, 32
question rows, 16 planted frames; top-k 1024 per (layer, query head), budget 64 units.

A step is one full retrieval (query prep, key scoring, top-k merge, votes and mass,
pool, max-min diversity, expansion) for one question against the resident index.
The metric is shallow keys scored per second: a key is one stored (layer, key head,
token) bf16 row of 256 bytes scored against its 7 query heads.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line. --impl reference times the CPU oracle (test infrastructure, the
only other code this script may run) on a bounded sample of the same workload.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "shallow keys scored/sec (1-h index retrieval)"
TRACE_EVERY = 8
MIN_KERNEL_LAUNCHES = 20       # score-kernel launches bracketed per run, at least
NOMINAL_HBM_GBS = 8000.0       # the GB300's nominal HBM3e bandwidth
SFU_EX2_PER_CLK_SM = 32        # ex2 results per clock per SM on the GB300 (measured 29.8)
UNIT = "keys/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="hour1")
    ap.add_argument("--cpu-frames", type=int, default=600,
                    help="frames of the stream the CPU oracle baseline scores")
    ap.add_argument("--ref-frames", type=int, default=100,
                    help="frames of the stream one reference-arm step scores")
    ap.add_argument("--frames", type=int, default=0,
                    help="truncate the stream to this many frames (small profiling case)")
    ap.add_argument("--sweep", action="store_true",
                    help="query latency versus history length (64 frames to 3 h), with and "
                         "without window compression; one JSON line per length")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    return ap.parse_args()


def dist_init(n_gpus: int):
    import torch
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(local)
    return rank, world, local


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = torch.device("cuda", torch.cuda.current_device()) if torch.cuda.is_available() else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_step_per_rank: int, steps: int, world: int,
                   max_ms_over_ranks: float) -> float:
    """Units per second of the whole job: every rank processes its own units (weak
    scaling), timed by the slowest rank."""
    return units_per_step_per_rank * steps * world / (max_ms_over_ranks / 1e3)


class ClockSampler:
    """nvidia-smi clock / throttle samples around the timed region. The sampler starts
    before the warm-up (so that nvidia-smi's start-up is not inside the region) and keeps
    the samples stamped within one sampling period of the region."""

    QUERY = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    PERIOD_S = 0.1

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines: list[str] = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", str(int(self.PERIOD_S * 1000))],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (OSError, ValueError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    @staticmethod
    def parse(lines: list[str], t0: float | None = None, t1: float | None = None,
              pad: float = 0.1) -> dict:
        """Median SM clock, max clock and active throttle reasons of the samples stamped
        in [t0 - pad, t1 + pad] (host epoch seconds), or of all samples if none is."""
        import datetime
        rows = []
        for ln in lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 10:
                continue
            try:
                ts = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                rows.append((ts, float(f[2]), float(f[3]), f[6:10]))
            except ValueError:
                continue
        inside = [r for r in rows if t0 is None or t0 - pad <= r[0] <= t1 + pad]
        use = inside or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = {nm for r in use for nm, v in zip(names, r[3]) if v.lower() == "active"}
        return {"sm_mhz": statistics.median(r[1] for r in use) if use else None,
                "sm_max_mhz": max(r[2] for r in use) if use else None,
                "reasons": sorted(reasons), "samples": len(use),
                "window": "timed region" if inside else "whole run"}

    def stop(self, t0: float | None = None, t1: float | None = None) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        return self.parse(self.lines, t0, t1, self.PERIOD_S)


def measured_peak_gbs() -> tuple[float, str]:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


CPU_BASELINE_SECONDS = 10.0


def cpu_baseline(w, data_keys_cpu, q_cpu, frames: int) -> dict:
    """The oracle as it stands, on the first `frames` frames of the stream."""
    import numpy as np
    from oracle import retrieval as R
    from paper_2609_02780_gb300 import synth
    kb = synth.bf16_bits(data_keys_cpu[:, :, : frames * w.tokens_per_frame])
    qb = synth.bf16_bits(q_cpu)
    # the sample's retrieval repeated until about CPU_BASELINE_SECONDS of CPU work
    reps = 0
    t0 = time.perf_counter()
    while True:
        R.retrieve(kb, qb, n_units=frames, tokens_per_unit=w.tokens_per_unit, k=w.k,
                   budget=w.budget, pool_mult=w.pool_mult, n_prev=w.n_prev)
        reps += 1
        dt = time.perf_counter() - t0
        if dt >= CPU_BASELINE_SECONDS:
            break
    keys = w.n_slabs * frames * w.tokens_per_frame
    return {"value": keys * reps / dt, "unit": UNIT, "cores": len(os.sched_getaffinity(0)),
            "kind": "oracle", "seconds": round(dt, 3), "repetitions": reps,
            "sample": f"oracle retrieve over the first {frames} of {w.n_frames} frames "
                      f"({keys} keys, all {w.n_layers} layers), fp64 numpy, {reps} times"}


def run_reference(args):
    """Reference arm: the CPU oracle on a bounded sample, per step."""
    import numpy as np
    import torch
    from paper_2609_02780_gb300 import synth
    from oracle import retrieval as R
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = synth.PRESETS[args.workload]
    frames = min(args.ref_frames, w.n_frames)
    sample = w.replace(n_frames=frames, n_planted=max(1, w.n_planted * frames // w.n_frames))
    data = synth.make_workload(sample, device="cpu")
    kb, qb = synth.bf16_bits(data["keys"]), synth.bf16_bits(data["q"])
    keys = sample.keys_per_query

    def step():
        R.retrieve(kb, qb, n_units=sample.n_units, tokens_per_unit=w.tokens_per_unit,
                   k=w.k, budget=w.budget, pool_mult=w.pool_mult, n_prev=w.n_prev)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    value = keys * args.steps / dt
    cores = len(os.sched_getaffinity(0))
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": {"workload": f"{w.name} first {frames} frames",
                       "keys_per_step": keys},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"first {frames} of {w.n_frames} frames per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# DRAM bytes of one k_score launch on the full 1-hour workload, from a 1-pass ncu
# capture of dram__bytes_read.sum + dram__bytes_write.sum; valid only for the kernel
# sources it was taken on (their sha256 below), reported as null otherwise.
TRAFFIC_RECORD = {"workload": "hour1",
                  "sources_sha256": "fb256876bb1813875b2b719fb668c6a680adc158037e18d811bb80b002fd174f",
                  "dram_bytes": 2891363584 + 23119872}  # read + write
SCORE_SOURCES = ("ss_score.cu", "ss_internal.cuh", "ss_device.cuh")


def score_sources_sha256() -> str:
    import hashlib
    h = hashlib.sha256()
    for f in SCORE_SOURCES:
        with open(os.path.join(ROOT, "paper_2609_02780_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def recorded_traffic(w) -> float | None:
    r = TRAFFIC_RECORD
    if r["dram_bytes"] is None or w.name != r["workload"] or w.window_frames:
        return None
    return float(r["dram_bytes"]) if score_sources_sha256() == r["sources_sha256"] else None


class host_call:
    """One ss_retrieve_host call through the C ABI with its arguments marshalled once
    (the call a C host makes; the Python binding's per-call bookkeeping stays out)."""

    def __init__(self, ss, idx, q_pin, p, ws, stream):
        import ctypes as C
        import torch
        self.lib = ss._abi.load()
        nexp = p.budget * (1 + p.n_prev)
        self.bufs = [torch.empty(n, dtype=torch.int32).pin_memory()
                     for n in (p.budget, nexp, nexp * idx.frames_per_unit, 4)]
        self.hr = ss._abi.HostResult(*[b.data_ptr() for b in self.bufs])
        self.pc = p.to_c()
        self.args = (idx.handle, C.c_void_p(q_pin.data_ptr()), C.c_int32(q_pin.shape[1]),
                     C.byref(self.pc), C.byref(self.hr), C.c_void_p(ws.data_ptr()),
                     C.c_size_t(ws.numel()), C.c_void_p(stream.cuda_stream))
        self._keep = (q_pin, ws)

    def __call__(self):
        st = self.lib.ss_retrieve_host(*self.args)
        if st != 0:
            raise RuntimeError(self.lib.ss_last_error().decode())

    def frames(self) -> list[int]:
        n = int(self.bufs[3][3])
        return self.bufs[2][:n].tolist()


def time_compress(ss, w, keys, dev, reps: int = 3) -> tuple[float, list[float]]:
    """Median device time of ss_index_compress over the whole stream (fresh indexes built
    from the same keys; a small compression first loads the kernel and its attributes)."""
    import torch
    warm = ss.Index(w.n_layers, w.n_q_heads, w.n_kv_heads, w.tokens_per_frame,
                    2 * w.window_frames, frames_per_unit=w.frames_per_unit, device=dev)
    warm.append(keys[:, :, : 2 * w.window_frames * w.tokens_per_frame])
    warm.compress(w.window_frames, n_centroids=w.n_centroids, iters=w.kmeans_iters)
    torch.cuda.synchronize(dev)
    times = []
    for _ in range(reps):
        ix = ss.Index(w.n_layers, w.n_q_heads, w.n_kv_heads, w.tokens_per_frame, w.n_frames,
                      frames_per_unit=w.frames_per_unit, device=dev)
        ix.append(keys)
        c0 = torch.cuda.Event(enable_timing=True)
        c1 = torch.cuda.Event(enable_timing=True)
        c0.record()
        ix.compress(w.window_frames, n_centroids=w.n_centroids, iters=w.kmeans_iters)
        c1.record()
        torch.cuda.synchronize(dev)
        times.append(c0.elapsed_time(c1))
        ix.close()
    return statistics.median(times), times


def host_copy_bytes(budget: int, nexp: int, frames_per_unit: int) -> int:
    """Bytes that ss_retrieve_host's kernels write into page-locked host memory per call,
    at most: the selection (K ids), the expansion and its frames (at most K (1 + n_prev)
    units, times frames per unit), the four counts and the status word."""
    return 4 * budget + 4 * nexp + 4 * nexp * frames_per_unit + 16 + 4


def run_ours(args):
    import numpy as np
    import torch
    import paper_2609_02780_gb300 as ss
    from paper_2609_02780_gb300 import synth

    rank, world, local = dist_init(args.gpus)
    dev = torch.device("cuda", local)
    w = synth.PRESETS[args.workload]
    if args.frames:
        w = w.replace(n_frames=args.frames,
                      n_planted=max(1, w.n_planted * args.frames // w.n_frames))
    n_streams = w.n_streams
    clusters = w.window_frames > 0
    fwd_I = int(w.extra.get("intermediate", 0))   # the question's forward (Eq. 10) too
    idxs, qs = [], []
    keys_cpu = q_cpu = None
    compress_ms = compress_all = None
    for st in range(n_streams):
        data = synth.make_workload(w, device=dev, stream=rank * n_streams + st)
        idx = ss.Index(w.n_layers, w.n_q_heads, w.n_kv_heads, w.tokens_per_frame, w.n_frames,
                       frames_per_unit=w.frames_per_unit, device=dev)
        idx.append(data["keys"])
        if fwd_I:
            idx.append_values(synth.make_values(w, device=dev, seed=data["seed"]))
        if clusters:
            compress_ms, compress_all = time_compress(ss, w, data["keys"], dev)
            idx.compress(w.window_frames, n_centroids=w.n_centroids, iters=w.kmeans_iters)
        if st == 0:
            if rank == 0 and not args.no_cpu_baseline and not fwd_I:
                frames = min(args.cpu_frames, w.n_frames)
                keys_cpu = data["keys"][:, :, : frames * w.tokens_per_frame].cpu()
            q_cpu = data["q"].cpu()
        idxs.append(idx)
        qs.append(data["q"])
        del data
    torch.cuda.synchronize(dev)
    torch.cuda.empty_cache()

    p = ss.RetrieveParams(k=w.k, budget=w.budget, pool_mult=w.pool_mult, n_prev=w.n_prev,
                          n_recent=w.n_recent, q_agg=w.q_agg, head_agg=w.head_agg,
                          use_clusters=int(clusters))
    outs = [ss.Result(ix, p) for ix in idxs]
    ws = torch.empty(ss.workspace_bytes(idxs, [q.shape[1] for q in qs], p),
                     dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    # The timed region runs the steps back to back. Events inside a step separate its
    # kernels (no programmatic overlap), so the score kernel is bracketed on every
    # TRACE_EVERY-th step only; per-step latency is taken in a second region after it,
    # and a third region brackets the score kernel on every one of its steps (at least
    # MIN_KERNEL_LAUNCHES launches in all).
    n_traced = (args.steps + TRACE_EVERY - 1) // TRACE_EVERY
    n_lat = min(max(args.steps, MIN_KERNEL_LAUNCHES), 50)
    n_kern = max(MIN_KERNEL_LAUNCHES, min(args.steps, 50))
    k_begin = [torch.cuda.Event(enable_timing=True) for _ in range(n_traced + n_kern)]
    k_end = [torch.cuda.Event(enable_timing=True) for _ in range(n_traced + n_kern)]
    s_begin = [torch.cuda.Event(enable_timing=True) for _ in range(n_lat)]
    s_end = [torch.cuda.Event(enable_timing=True) for _ in range(n_lat)]
    for ev in k_begin + k_end:
        ev.record(stream)  # create the events before handing them to the library

    fw = None
    if fwd_I:
        # the question's forward through the shallow layers produces the query rows the
        # retrieval scores (one stream per GPU)
        fw_layers = synth.make_forward_weights(w, fwd_I, device=dev)
        fw_h = synth.make_question_rows(w, device=dev)
        fw_p = ss.ForwardParams(fwd_I)
        fw_q = torch.empty_like(qs[0])
        fw_hout = torch.empty(w.n_rows, w.n_q_heads * 128, dtype=torch.float32, device=dev)
        fw_ws = torch.empty(idxs[0].forward_workspace_bytes(w.n_rows, fw_p), dtype=torch.uint8,
                            device=dev)
        fw_status = torch.zeros(1, dtype=torch.int32, device=dev)
        fw_bytes = (sum(t.numel() * 2 for L in fw_layers for t in L.values() if t is not None) +
                    2 * w.key_bytes)

        def forward():
            idxs[0].forward(fw_layers, fw_h, fw_p, q_out=fw_q, h_out=fw_hout, workspace=fw_ws,
                            status=fw_status)
        qs = [fw_q]
        fw = {"bytes": fw_bytes, "ms": []}

    def step(tr=None):
        if fw is not None:
            forward()
        ss.retrieve_batched(idxs, qs, p, outs=outs, workspace=ws, trace=tr)

    clocks = ClockSampler(local)
    clocks.start()
    for _ in range(max(3, args.warmup)):
        step()
    for o in outs:
        o.check()
    barrier(world)
    torch.cuda.synchronize(dev)
    wall0 = time.time()
    t_all0 = torch.cuda.Event(enable_timing=True)
    t_all1 = torch.cuda.Event(enable_timing=True)
    t_all0.record(stream)
    for i in range(args.steps):
        j = i // TRACE_EVERY
        step((k_begin[j], k_end[j]) if i % TRACE_EVERY == 0 else None)
    t_all1.record(stream)
    torch.cuda.synchronize(dev)
    wall1 = time.time()
    barrier(world)
    for i in range(n_lat):
        s_begin[i].record(stream)
        step()
        s_end[i].record(stream)
    for j in range(n_traced, n_traced + n_kern):
        step((k_begin[j], k_end[j]))
    if fw is not None:
        # the forward alone, bracketed on each of n_kern calls
        f_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                for _ in range(n_kern)]
        for a, b in f_ev:
            a.record(stream)
            forward()
            b.record(stream)
        torch.cuda.synchronize(dev)
        fw["ms"] = [a.elapsed_time(b) for a, b in f_ev]
        if int(fw_status.item()) != 0:
            raise RuntimeError(f"forward status {int(fw_status.item())}")
    torch.cuda.synchronize(dev)
    clk = clocks.stop(wall0, wall1)
    for o in outs:
        o.check()
    total_ms = t_all0.elapsed_time(t_all1)
    total_ms = max_over_ranks(total_ms, world)
    step_ms = sorted(s_begin[i].elapsed_time(s_end[i]) for i in range(n_lat))
    k1_ms = [k_begin[j].elapsed_time(k_end[j]) for j in range(n_traced + n_kern)]
    keys = w.keys_per_query * n_streams
    value = whole_job_rate(keys, args.steps, world, total_ms)

    # end to end through the C ABI's host entry point: the question's rows in pinned host
    # memory, the selection back in host memory, both copies inside the timed region
    e2e = None
    if not args.no_e2e and n_streams == 1 and fw is None:
        idx = idxs[0]
        q_pin = q_cpu.pin_memory()
        call = host_call(ss, idx, q_pin, p, ws, stream)
        for _ in range(3):
            call()
        barrier(world)
        t0 = time.perf_counter()
        for _ in range(args.steps):
            call()
        dt = max_over_ranks(time.perf_counter() - t0, world)
        got = idx.retrieve_host(q_pin, p, workspace=ws)   # the Python binding agrees
        assert got["frames"] == call.frames(), "host entry point results differ"
        nexp = p.budget * (1 + p.n_prev)
        e2e = {"value": keys * args.steps * world / dt, "unit": UNIT,
               # the kernels read only the rows the path needs from the page-locked
               # question (the last one of each layer under the default LAST reading)
               "h2d_bytes_per_step": int(q_pin.numel() * 2 // (q_pin.shape[1] if p.q_agg == 0 else 1)),
               "d2h_bytes_per_step": host_copy_bytes(p.budget, nexp, w.frames_per_unit),
               "ms_per_step": dt / args.steps * 1e3}

    if rank != 0:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return
    peak, peak_kind = measured_peak_gbs()
    k1_avg_s = statistics.mean(k1_ms) / 1e3
    if clusters:
        # the scoring stage reads the centroids of every window of every slab
        n_cand = w.n_slabs * (w.n_frames // w.window_frames) * w.n_centroids * n_streams
        alg_bytes = n_cand * 256
        kernel = "k_dense"
        launches = 9   # k_sample, k_cluster_map, k_dense, k_select, k_centroid_weight,
        #                k_mass, k_pool, k_gram, k_maxmin
    elif w.q_agg == 2:
        # every question row attends: two passes over the keys (statistics, weights)
        alg_bytes = 2 * keys * 256
        kernel = "k_rm_stats + k_rm_combine + k_rm_alpha"
        launches = 9   # k_sample, the three passes, k_select, k_mass_general, k_pool,
        #                k_gram, k_maxmin
    else:
        alg_bytes = keys * 256
        kernel = "k_score"
        launches = 7   # k_sample, k_score, k_select, k_mass, k_pool, k_gram, k_maxmin
    achieved = alg_bytes / k1_avg_s / 1e9
    roof = None
    if w.q_agg == 2 and fw is None:
        # every key's score is exponentiated once per question row in each pass; at the
        # GB300's ex2 rate that takes ~0.6 of the two key reads' HBM time, so HBM bounds
        # the three kernels (the ex2 rate is reported beside it)
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        clk_mhz = clk.get("sm_max_mhz") or 2070.0
        ex2_peak = SFU_EX2_PER_CLK_SM * sms * clk_mhz * 1e6 / 1e9          # G ex2/s
        G = w.n_q_heads // w.n_kv_heads
        n_ex2 = 2 * keys * G * w.n_rows                                     # both passes
        roof = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": None,
                "frac_nominal": achieved / NOMINAL_HBM_GBS, "kernel": kernel,
                "peak_kind": peak_kind, "algorithmic_bytes_per_launch": alg_bytes,
                "ex2": {"achieved": n_ex2 / k1_avg_s / 1e9, "peak": ex2_peak, "unit": "Gex2/s",
                        "frac": n_ex2 / k1_avg_s / 1e9 / ex2_peak,
                        "peak_kind": f"derived: {SFU_EX2_PER_CLK_SM} ex2/clk/SM x {sms} SMs x "
                                     f"{clk_mhz:.0f} MHz",
                        "algorithmic_ex2_per_launch": n_ex2}}
    if fw is not None:
        # the forward dominates the step: every layer's weights and stored keys and values
        # read once per question
        k1_avg_s = statistics.mean(fw["ms"]) / 1e3
        alg_bytes = fw["bytes"]
        # per layer: 2 norms, 4 projections, q/k/v, attention, merge, and SwiGLU unless the
        # gate/up projection runs as one K split (2 I / 128 tiles above two per SM) and
        # applies it in its epilogue
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        fused = (2 * sms) // (2 * fwd_I // 128) <= 1
        kernel = ("question forward (k_fw_norm_row, k_fw_gemm, k_fw_qkv, k_fw_attn, "
                  "k_fw_attn_out" + ("" if fused else ", k_fw_swiglu") + ")")
        launches += 2 + (9 if fused else 10) * w.n_layers   # RoPE table, final residual
        achieved = alg_bytes / k1_avg_s / 1e9
    traffic = recorded_traffic(w) if not args.frames and n_streams == 1 and fw is None else None
    if roof is None:
        roof = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": traffic,
                "frac_nominal": achieved / NOMINAL_HBM_GBS,
                "kernel": kernel, "peak_kind": peak_kind,
                "algorithmic_bytes_per_launch": alg_bytes}
    cpu = None
    if keys_cpu is not None:
        cpu = cpu_baseline(w, keys_cpu, q_cpu, keys_cpu.shape[2] // w.tokens_per_frame)
    desc = (f"{w.name}: {w.n_layers} layers x {w.n_kv_heads} kv heads x "
            f"{w.n_frames} frames x {w.tokens_per_frame} tokens, Hq {w.n_q_heads}, "
            f"R {w.n_rows}, k {w.k}, budget {w.budget}, pool {w.pool_mult * w.budget}")
    if n_streams > 1:
        desc += f", {n_streams} streams per GPU in one batched call"
    if fw is not None:
        desc += (f", question forward through {w.n_layers} synthetic decoder layers (hidden "
                 f"{w.n_q_heads * 128}, MLP {fwd_I}) attending to the stored keys and values, "
                 f"then retrieval on its query rows")
    if clusters:
        desc += (f", windows of {w.window_frames} frames compressed to {w.n_centroids} "
                 f"centroids ({w.kmeans_iters} Lloyd rounds), retrieval over centroids")
    config = {"workload": desc, "keys_per_step": keys, "index_bytes": w.key_bytes * n_streams,
              "l2": f"inputs larger than L2 ({w.key_bytes * n_streams / 1e9:.2f} GB index vs "
                    f"129 MB L2), no flush",
              "parallelism": f"replicas x{world} (independent streams per GPU)"}
    if fw is not None:
        config["forward_ms"] = statistics.mean(fw["ms"])
        config["forward_bytes"] = fw["bytes"]
        config["index_bytes"] = 2 * w.key_bytes
    if clusters:
        config["compress_ms"] = compress_ms
        config["compress_ms_all"] = compress_all
        config["candidates_per_step"] = n_cand
        config["l2"] = (f"{alg_bytes / 1e6:.1f} MB of centroids per step: below L2, so the "
                        f"timed steps read them from L2 (no flush)")
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": max(3, args.warmup),
        "ms_per_step": total_ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": config,
        "latency_ms": {"p50": statistics.median(step_ms),
                       "p90": step_ms[min(len(step_ms) - 1, int(0.9 * len(step_ms)))],
                       "steps": n_lat,
                       "score_kernel_avg": statistics.mean(k1_ms),
                       "score_kernel_p50": statistics.median(k1_ms),
                       "score_kernel_launches_timed": len(k1_ms)},
        "roofline": roof,
        "clocks": clk,
        "gpu_launches": launches * args.steps,
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


SWEEP_FRAMES = (64, 128, 256, 512, 1024, 1800, 3600, 7200, 10800)


def run_sweep(args):
    """Query-time latency of one retrieval versus the length of the retained history (the
    1-hour stream's shape at 1 fps: 64 frames to 3 hours), without compression (every key
    scored) and with the history's 20-frame windows compressed to 64 centroids except the
    latest 60 frames (LC-on: centroids and the recent raw tail scored). Device time of
    the retrieval with CUDA events, p50 of the timed steps."""
    import torch
    import paper_2609_02780_gb300 as ss
    from paper_2609_02780_gb300 import synth
    dev = torch.device("cuda", 0)
    base = synth.PRESETS["hour1"]
    steps = max(10, args.steps)

    def p50(fn):
        for _ in range(3):
            fn()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(steps)]
        for a, b in ev:
            a.record()
            fn()
            b.record()
        torch.cuda.synchronize(dev)
        return statistics.median(a.elapsed_time(b) for a, b in ev)

    for frames in SWEEP_FRAMES:
        w = base.replace(n_frames=frames, n_planted=max(1, min(16, frames // 64)))
        data = synth.make_workload(w, device=dev)
        idx = ss.Index(w.n_layers, w.n_q_heads, w.n_kv_heads, w.tokens_per_frame, frames,
                       device=dev)
        idx.append(data["keys"])
        p = ss.RetrieveParams(k=w.k, budget=w.budget)
        res = ss.Result(idx, p)
        ws = torch.empty(idx.workspace_bytes(w.n_rows, p), dtype=torch.uint8, device=dev)
        q = data["q"]
        off = p50(lambda: idx.retrieve(q, k=p.k, budget=p.budget, out=res, workspace=ws))
        on = None
        n_comp = (max(0, frames - 60) // 20) * 20
        if n_comp:
            idx.compress(20, n_centroids=64, iters=5, first_frame=0, n_frames=n_comp)
            pc = ss.RetrieveParams(k=512, budget=w.budget, use_clusters=1)
            rc = ss.Result(idx, pc)
            wc = torch.empty(idx.workspace_bytes(w.n_rows, pc), dtype=torch.uint8, device=dev)
            on = p50(lambda: idx.retrieve(q, k=pc.k, budget=pc.budget, use_clusters=1, out=rc,
                                          workspace=wc))
        # LC-on with the paper's compression: units older than the latest 60 leave the
        # detailed window into online clusters (tau 0.9); a question is answered by token
        # voting over the detailed units plus the top-8 clusters (Eq. 13)
        del idx, res, ws
        torch.cuda.empty_cache()
        on_units = None
        if frames > 60:
            ix2 = ss.Index(w.n_layers, w.n_q_heads, w.n_kv_heads, w.tokens_per_frame, frames,
                           device=dev)
            ix2.append(data["keys"])
            n_leave = ix2.units_over_budget(0, 60)
            ix2.cluster_units(n_leave, 0.9, max_clusters=min(frames, 16384))
            r2 = ss.Result(ix2, p)
            w2 = torch.empty(ix2.workspace_bytes(w.n_rows, p), dtype=torch.uint8, device=dev)

            def both():
                ix2.retrieve(q, k=p.k, budget=p.budget, out=r2, workspace=w2)
                ix2.select_clusters(q, k_l=8)
            on_units = p50(both)
            n_clusters = int(ix2.unit_clusters()["sizes"].numel())
            del ix2, r2, w2
            torch.cuda.empty_cache()
        keys = w.keys_per_query
        print(json.dumps({"sweep": "query latency vs history", "frames": frames,
                          "hours": round(frames / 3600, 3), "keys": keys,
                          "index_bytes": w.key_bytes, "lc_off_ms": off,
                          "lc_off_keys_per_s": keys / (off / 1e3),
                          "lc_on_ms": on, "lc_on_compressed_frames": n_comp,
                          "lc_units_ms": on_units,
                          "lc_units_clusters": n_clusters if on_units is not None else None}),
              flush=True)
        del data
        torch.cuda.empty_cache()


def main():
    args = parse()
    if args.sweep:
        run_sweep(args)
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
