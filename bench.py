#!/usr/bin/env python
"""Benchmark of the ReSpec verify-and-draft step on GB300.

A step is one pass of the whole hot path over one batch: rs_entropy_gate ->
rs_match_scan -> rs_tree_verify_attn (one layer) -> rs_accept, on one stream,
replayed from a CUDA graph.  Metric: steps/s (whole job), plus the KV +
logits HBM bytes per step as GB/s and as a fraction of the measured peak.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the fp64 CPU oracle, timed on a sample
  python bench.py --retrieval            # linear scan vs inverted index on long buffers

Under torchrun each rank runs its own batch (requests are independent: weak
scaling, no data-path collective); the timed region is bracketed by a barrier
and a device synchronise on every rank and the slowest rank's time is used.
Rank 0 prints one JSON line.
"""
import argparse
import hashlib
import re
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tree-verify steps/s and KV+logits HBM GB/s (fraction of GB300 peak), 1 GPU"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
WORKLOAD_TEXT = {
    "tiny": "Tiny: B=1, Hq=Hkv=4, D=64, S=256, N=9, V=1024",
    "7b": "7B-shape: B=1, Hq=Hkv=32, D=128, S=2048, N=41, V=32000",
    "gqa16k": "8B-GQA long context: B=1, Hq=32, Hkv=8, D=128, S=16384, N=145, V=128256",
    "batched": "Batched serving: B=16, Hq=32, Hkv=8, D=128, S~U[1024,8192], N=25-65, V=128256",
    "13b32k": "13B-shape long context: B=4, Hq=Hkv=40, D=128, S=32768, N=65, V=32000",
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", default="13b32k", choices=sorted(WORKLOAD_TEXT))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-budget-s", type=float, default=12.0,
                    help="seconds of oracle attention work in the CPU baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true",
                    help="skip the end-to-end (host buffers) measurement: lean runs for profiling")
    ap.add_argument("--requests", type=int, default=0,
                    help="keep only the first N requests of the workload (small profiling cases)")
    ap.add_argument("--soak-s", type=float, default=1.0,
                    help="seconds of untimed step replays right before the timed steps, so that the "
                         "sampled SM clocks cover the GPU under load")
    ap.add_argument("--retrieval", action="store_true",
                    help="instead of the step: rs_match_scan against the inverted index "
                         "(rs_match_index_*) on long synthetic buffers, one JSON line per length")
    ap.add_argument("--lengths", default="32768,262144,1048576,4194304",
                    help="buffer lengths per request for --retrieval")
    return ap.parse_args()


# ------------------------------------------------------------------ ranks
def rank_seed(seed, rank):
    """Each rank draws its own batch (requests are independent: weak scaling)."""
    return seed + 7919 * rank


def slowest(value, dist, device):
    """Max over ranks of a per-rank duration (identity without a process group)."""
    if dist is None:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(steps_per_rank, world, seconds):
    """Whole-job throughput: every rank's steps over the slowest rank's time."""
    return steps_per_rank * world / seconds


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi samples every 200 ms while running (read-only queries)."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.rows = []
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.Q, "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                self.rows.append(parts)

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=5)

    def summary(self):
        if not self.rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in self.rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in self.rows:
            for n, val in zip(names, r[5:9]):
                if val.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(self.rows)}


# ------------------------------------------------------------------ bytes
def algorithmic_bytes(w):
    s = w.spec
    R = w.R
    kv_rows = int((w.ctx_len.astype(int) + w.node_off[1:] - w.node_off[:-1]).sum())
    attn = 2 * kv_rows * s.Hkv * s.D * 2 + R * s.Hq * s.D * 2 + R * s.Hq * (s.D + 1) * 4
    logits = R * s.V * 4
    tokens = int(w.tok_off[-1]) * 4
    return dict(attn=attn, kv=2 * kv_rows * s.Hkv * s.D * 2, logits=logits, tokens=tokens,
                step=attn + logits + 2 * tokens,
                flops=4 * int(sum((w.node_off[b + 1] - w.node_off[b]) * (w.ctx_len[b] + w.node_off[b + 1] - w.node_off[b])
                                  for b in range(w.B))) * s.Hq * s.D)


def attn_source_sha():
    """Hash of the attention kernels' sources with comments and blank space
    taken out, so that a comment edit keeps the committed traffic records
    while any change to the code retires them."""
    h = hashlib.sha256()
    for f in ("attn.cu", "attn_core.cuh", "attn_pair.cuh", "sm100.cuh"):
        with open(os.path.join(ROOT, "paper_2511_01282_gb300", "csrc", f)) as fh:
            src = fh.read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)   # block comments
        src = re.sub(r"//[^\n]*", " ", src)                # line comments
        h.update(" ".join(src.split()).encode())
    return h.hexdigest()[:16]


def committed_traffic(workload):
    """DRAM bytes per attention launch from a committed ncu summary, if it was
    taken on the current kernel source; else None."""
    path = os.path.join(ROOT, "profiles", "attn_traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f)
    e = d.get(workload)
    if not e or e.get("source_sha") != attn_source_sha():
        return None
    return e.get("dram_bytes_per_launch")


def attn_roofline(by, attn_s, gbs, hbm, peaks, peak_kind, launch_ms, traffic):
    """The attention call against the bound its arithmetic sets: HBM when its
    bytes at the copy bandwidth take longer than its FLOPs at the bf16 tensor
    rate, the tensor cores otherwise (the burst figure: the call is timed
    alone).  Both rates are reported either way."""
    tc_burst = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    tc_sust = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    tflops = by["flops"] / attn_s / 1e12
    tensor = by["flops"] / (tc_burst * 1e12) > by["attn"] / (hbm * 1e9)
    r = {"kernel": "rs_tree_verify_attn (prep + main + combine)", "bound": "tensor" if tensor else "hbm",
         "achieved": tflops if tensor else gbs, "peak": tc_burst if tensor else hbm,
         "unit": "TFLOP/s" if tensor else "GB/s", "frac": tflops / tc_burst if tensor else gbs / hbm,
         "peak_kind": peak_kind, "algorithmic_bytes_per_launch": by["attn"],
         "algorithmic_flops_per_launch": by["flops"], "launch_ms": launch_ms, "traffic": traffic,
         "gbs": gbs, "gbs_frac": gbs / hbm, "tflops": tflops, "tflops_frac_sustained": tflops / tc_sust}
    if tensor:
        r["peak_note"] = "bf16 burst (the call is timed alone); tflops_frac_sustained against the sustained rate"
    return r


# ------------------------------------------------------------------ end to end
def end_to_end(st, st2, graph, stream, K, W, barrier):
    """K steps from pinned host inputs to decisions on the host, through the
    same calls.  Two device copies of the inputs (st, st2: one pinned host
    buffer) alternate, so the upload of step i + 1 (copy engine) overlaps step
    i's kernels; the host holds step i - 1's decisions before it enqueues
    step i + 1.  Returns (seconds, h2d bytes per step, d2h bytes per step)."""
    import torch
    st2.prime()
    torch.cuda.synchronize()
    for _ in range(2):
        st2.step(stream)
    torch.cuda.synchronize()
    graph2 = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph2, stream=stream):
        st2.step(stream)
    sets = [(st, graph, st.result_buffers()), (st2, graph2, st2.result_buffers())]
    copy_stream = torch.cuda.Stream()

    def e2e_step(i, done):
        x = i & 1
        sx, gx, bx = sets[x]
        if done[x] is not None:  # step i - 2 has finished with this input set
            copy_stream.wait_event(done[x])
        h = sx.upload(copy_stream)
        up = torch.cuda.Event()
        up.record(copy_stream)
        stream.wait_event(up)
        with torch.cuda.stream(stream):
            gx.replay()
        d = sx.download_into(bx, stream)
        ev = torch.cuda.Event()
        ev.record(stream)
        done[x] = ev
        if i >= 1:  # step i - 1's decisions are on the host
            done[x ^ 1].synchronize()
        return h, d

    done = [None, None]
    for i in range(max(W, 2)):
        e2e_step(i, done)
    torch.cuda.synchronize()
    barrier()
    done = [None, None]
    t0 = time.perf_counter()
    h2d = d2h = 0
    for i in range(K):
        h2d, d2h = e2e_step(i, done)
    torch.cuda.synchronize()
    return time.perf_counter() - t0, h2d, d2h


# ------------------------------------------------------------------ CPU oracle sample
def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def oracle_attn_rows(w, rows, workers):
    """The oracle's attention on the given (node, head) rows, split into
    disjoint row chunks run by `workers` host threads (the oracle's C code
    releases the GIL; each row is computed on its own, so the split leaves its
    arithmetic unchanged)."""
    import concurrent.futures as cf

    import numpy as np

    import oracle
    s = w.spec
    rr = np.asarray(rows, dtype=np.int64).reshape(-1, 2)
    if workers <= 1 or len(rr) < 2:
        oracle.tree_attn(w.q, w.k, w.v, w.kv_off, w.ctx_len, w.node_off, w.parents, s.Hq, s.Hkv, s.D,
                         s.D ** -0.5, rows=rr)
        return
    parts = np.array_split(rr, min(len(rr), workers * 4))
    with cf.ThreadPoolExecutor(max_workers=workers) as ex:
        list(ex.map(lambda part: oracle.tree_attn(w.q, w.k, w.v, w.kv_off, w.ctx_len, w.node_off, w.parents,
                                                  s.Hq, s.Hkv, s.D, s.D ** -0.5, rows=part), parts))


def oracle_entropy_rows(w, workers):
    import concurrent.futures as cf

    import numpy as np

    import oracle
    if workers <= 1:
        return oracle.entropy_rows(w.logits)
    parts = np.array_split(np.arange(w.R), min(w.R, workers))
    with cf.ThreadPoolExecutor(max_workers=workers) as ex:
        res = list(ex.map(lambda ix: oracle.entropy_rows(w.logits[ix[0]:ix[-1] + 1]) if len(ix) else
                          np.zeros(0), parts))
    return np.concatenate(res)


def oracle_step_sample(w, budget_s, workers=1, rows_cache={}):
    """Time the oracle on a bounded sample of one step on `workers` host
    threads.  Entropy (rows split over the threads), gate, scan and accept run
    over the whole batch; the attention runs on as many (node, head) rows of
    request 0 as fit the budget and is scaled to all rows.  Returns (estimated
    seconds per step, sample text, extrapolation record)."""
    import numpy as np

    import oracle
    s = w.spec
    f32 = lambda x: float(np.float32(x))  # noqa: E731
    t = time.perf_counter()
    H = oracle_entropy_rows(w, workers)
    oracle.gate(H, w.node_off, w.row_commit, w.hist, w.hist_n, s.l, f32(s.lambda_e), f32(s.theta_entropy))
    oracle.match_scan(w.tokens, w.tok_off, w.k_star_hint, w.scores, f32(s.theta_score), s.top_c, s.chain_len,
                      s.pos_cap)
    oracle.accept(w.logits, w.node_off, w.tree_tokens, w.parents, w.source, w.chain, w.sel_pos, w.tok_off,
                  w.scores, s.beta, f32(s.tau), s.phi, s.m, f32(s.alpha), 64)
    t_rest = time.perf_counter() - t
    # attention on (node, head) rows of request 0, as many as fit the budget
    n0, n1 = int(w.node_off[0]), int(w.node_off[1])
    total_rows = w.R * s.Hq
    key = (id(w), budget_s, workers)
    if key not in rows_cache:
        t1 = time.perf_counter()
        oracle_attn_rows(w, [(n0, 0)], 1)
        per_row = max(time.perf_counter() - t1, 1e-6)
        rows_cache[key] = max(1, min(int(budget_s * workers / per_row), (n1 - n0) * s.Hq, total_rows))
    nrows = rows_cache[key]
    rows = [(n0 + (i % (n1 - n0)), (i // (n1 - n0)) % s.Hq) for i in range(nrows)]
    t = time.perf_counter()
    oracle_attn_rows(w, rows, workers)
    t_attn = time.perf_counter() - t
    scale = total_rows / float(nrows)
    est = t_rest + t_attn * scale
    text = ("oracle on %d host thread(s): entropy+gate+scan+accept over the whole batch (%.2f s) + attention "
            "on %d of %d (node, head) rows (%.2f s), attention scaled by %.1fx"
            % (workers, t_rest, nrows, total_rows, t_attn, scale))
    extra = {"rows_timed": nrows, "rows_total": total_rows, "scale": scale, "what": "attention rows",
             "measured_s": t_rest + t_attn, "estimated_s": est}
    return est, text, extra


# ------------------------------------------------------------------ reference arm
def run_reference(args, rank, world):
    if rank != 0:
        return 0
    import synth
    w = synth.make(args.workload, args.seed)
    cores = host_cores()
    ests = []
    text, extra = "", {}
    warm = min(args.warmup, 1)
    # keep the whole run to a couple of minutes whatever K is
    budget = max(0.05, min(1.5, 90.0 / max(args.steps + warm, 1)))
    t0 = time.perf_counter()
    for i in range(warm + args.steps):
        est, text, extra = oracle_step_sample(w, budget_s=budget, workers=cores)
        if i >= warm:
            ests.append(est)
    wall = time.perf_counter() - t0
    est = statistics.median(ests)
    value = 1.0 / est
    text += "; median of %d timed samples after %d untimed one(s)" % (args.steps, warm)
    extra = dict(extra, samples=args.steps, wall_s=wall)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": est * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD_TEXT[args.workload], "name": args.workload},
        "extrapolated": extra,
        "cpu_baseline": {"value": value, "unit": "steps/s", "cores": cores, "kind": "oracle", "sample": text,
                         "extrapolated": extra},
        "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ our arm
def run_ours(args, rank, world, local_rank):
    import numpy as np  # noqa: F401
    import torch

    import __graft_entry__
    import synth
    from paper_2511_01282_gb300 import respec as rs
    from paper_2511_01282_gb300.pipeline import VerifyStep, arrays_from_workload

    __graft_entry__.build()
    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
    spec = synth.CONFIGS[args.workload]
    if args.requests:
        import dataclasses
        spec = dataclasses.replace(spec, B=min(args.requests, spec.B))
    w = synth.build(spec, seed=rank_seed(args.seed, rank))
    s = w.spec
    p = rs.params(**s.params())
    st = VerifyStep(arrays_from_workload(w), p, s.Hq, s.Hkv, s.D, pos_cap=s.pos_cap, pinned_host=True)
    stream = torch.cuda.Stream()
    K, W = args.steps, args.warmup

    # row entropies for the first fused step, launches per step, then warm-up
    st.prime()
    torch.cuda.synchronize()
    n0 = rs.rs_launch_count()
    st.step(stream)
    torch.cuda.synchronize()
    launches_per_step = rs.rs_launch_count() - n0
    for _ in range(W):
        st.step(stream)
    torch.cuda.synchronize()

    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        st.step(stream)

    # L2 flush before every timed step and call: a read of a buffer twice the
    # L2 size evicts whatever the previous step or call left in the L2 and
    # writes its dirty lines back, outside the timed region (a write-only
    # flush would leave ~L2-size dirty lines for the timed work to write back)
    by = algorithmic_bytes(w)
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    l2 = int(getattr(props, "L2_cache_size", 0) or (126 << 20))
    flush_buf = torch.ones(2 * l2 // 4, dtype=torch.int32, device="cuda")
    flush_sink = torch.empty((), dtype=torch.int32, device="cuda")

    def flush():
        torch.amax(flush_buf, dim=0, out=flush_sink)

    def timed_replays(g, n):
        """Device milliseconds of n replays of graph g on the timed stream,
        each after an L2 flush that lies outside its pair of events."""
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
        with torch.cuda.stream(stream):
            for a, b in ev:
                flush()
                a.record(stream)
                g.replay()
                b.record(stream)
        torch.cuda.synchronize()
        return sum(a.elapsed_time(b) for a, b in ev)

    with torch.cuda.stream(stream):
        for _ in range(max(W, 3)):
            flush()
            graph.replay()
    torch.cuda.synchronize()

    clocks = ClockSampler(local_rank)
    clocks.start()

    def barrier():
        if dist is not None:
            dist.barrier()

    # ---- soak: untimed replays so the clock samples see the GPU under load
    t_soak = time.perf_counter()
    n_soak = 0
    while time.perf_counter() - t_soak < args.soak_s:
        with torch.cuda.stream(stream):
            for _ in range(20):
                flush()
                graph.replay()
        torch.cuda.synchronize()
        n_soak += 20

    # ---- timed region: K graph replays, each after an L2 flush
    barrier()
    torch.cuda.synchronize()
    local_ms = timed_replays(graph, K)
    barrier()
    t_ms = slowest(local_ms, dist, "cuda")
    ms_per_step = t_ms / K
    value = job_rate(K, world, t_ms / 1e3)

    # ---- per-call device time: a CUDA graph of one call, replayed n times on
    # the timed stream, each replay after an L2 flush (cold, as in the step)
    def time_call(fn, n):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn(stream)
        with torch.cuda.stream(stream):
            g.replay()  # warm
        torch.cuda.synchronize()
        return timed_replays(g, n) / n

    n_call = max(10, min(K, 50))
    call_ms = {"gate_rows": time_call(st.gate_rows, n_call),
               "scan": time_call(lambda sm: st.scan(stream=sm), n_call),
               "attn": time_call(st.attn, n_call), "accept": time_call(lambda sm: st.accept(stream=sm), n_call),
               "gate_from_logits": time_call(st.gate, n_call),
               "tree_sample": time_call(lambda sm: st.tree_sample(1.0, sm), n_call)}
    # retrieval from the inverted index (NEXT-4) on the same buffers
    st.build_index()
    call_ms["scan_indexed"] = time_call(lambda sm: st.scan(stream=sm, indexed=True), n_call)
    call_ms["index_build"] = time_call(st.build_index, 3)
    st.reset_state()
    torch.cuda.synchronize()

    # ---- end to end: pinned host inputs -> step -> decisions back to the host
    if args.no_e2e:
        K_e2e = 0
    else:
        K_e2e = K
        st2 = VerifyStep(arrays_from_workload(w), p, s.Hq, s.Hkv, s.D, pos_cap=s.pos_cap, host_blob=st.pinned_blob)
        e2e_s, h2d, d2h = end_to_end(st, st2, graph, stream, K, W, barrier)
        e2e_s = slowest(e2e_s, dist, "cuda")
    clocks.stop()

    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))

    def roof(name, nbytes, ms, what):
        gbs = nbytes / (ms / 1e3) / 1e9
        return {"kernel": name, "bound": "hbm", "achieved": gbs, "peak": hbm, "unit": "GB/s", "frac": gbs / hbm,
                "peak_kind": peak_kind, "algorithmic_bytes_per_launch": nbytes, "launch_ms": ms,
                "timing": "cold: L2 flushed before each call; " + what}

    attn_s = call_ms["attn"] / 1e3
    achieved = by["attn"] / attn_s / 1e9
    step_gbs = (by["kv"] + by["logits"]) / (ms_per_step / 1e3) / 1e9
    R, V = w.R, s.V
    small_acc = R * (4 + 4 * s.beta + 4 + 4 + 4 + 4 + 1) + w.B * (4 * 4 + 64 * 4)
    line = {
        "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16+f32", "data": "synthetic",
        "config": {"workload": WORKLOAD_TEXT[args.workload] + (" (first %d requests)" % s.B if args.requests else ""),
                   "name": args.workload, "batch_per_gpu": s.B,
                   "l2": ("flushed: each timed step and each timed call follows a read of a %.0f MB buffer "
                          "(twice the L2), outside its events; the step moves %.3f GB of KV + logits"
                          % (2 * l2 / 2**20, (by["kv"] + by["logits"]) / 1e9)),
                   "graph": "each step replays one CUDA graph of the 4 calls",
                   "step": "trigger on the row entropies rs_accept computed over the previous step's "
                           "verify logits (logits read once per step)"},
        "kv_logits_hbm": {"gbs": step_gbs, "frac": step_gbs / hbm, "peak": hbm, "peak_kind": peak_kind,
                          "bytes_per_step": by["kv"] + by["logits"],
                          "note": "every byte comes from HBM: the L2 is flushed before each step"},
        "roofline": attn_roofline(by, attn_s, achieved, hbm, peaks, peak_kind, call_ms["attn"],
                                  committed_traffic(args.workload)),
        "rooflines": {
            "accept": roof("rs_accept (logits row pass + decisions)", R * V * 4 + small_acc, call_ms["accept"],
                           "the whole call: row pass, and the decision kernel after it"),
            "gate_from_logits": roof("rs_entropy_gate (logits row pass + history push)", R * V * 4,
                                     call_ms["gate_from_logits"], "the whole call from the logits"),
            "tree_sample": roof("rs_tree_sample (logits row pass + draws + walk)", R * V * 4,
                                call_ms["tree_sample"], "the whole call"),
        },
        "call_ms": call_ms,
        "e2e": ({"value": job_rate(K, world, e2e_s), "unit": "steps/s", "h2d_bytes_per_step": h2d,
                 "d2h_bytes_per_step": d2h} if K_e2e else None),
        "gpu_launches": launches_per_step * K,
        "launches_per_step": launches_per_step,
        "clocks": dict(clocks.summary(), window="%.1f s soak of %d flushed step replays, then the timed steps, "
                       "the per-call timings and the end-to-end loop" % (args.soak_s, n_soak)),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cores = host_cores()
        est, text, extra = oracle_step_sample(w, budget_s=args.cpu_budget_s, workers=cores)
        est1, text1, extra1 = oracle_step_sample(w, budget_s=args.cpu_budget_s, workers=1)
        line["cpu_baseline"] = {"value": 1.0 / est, "unit": "steps/s", "cores": cores, "kind": "oracle",
                                "sample": text, "extrapolated": extra,
                                "one_core": {"value": 1.0 / est1, "unit": "steps/s", "cores": 1, "sample": text1,
                                             "extrapolated": extra1}}
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ retrieval leg
def run_retrieval(args):
    """rs_match_scan (O(t) per query) against rs_match_scan_indexed
    (O(occurrences of the key's last token) per query, after an O(t)
    rs_match_index_build) on long synthetic buffers: V = 32000, segments of
    8-64 tokens of which 30 % copy an earlier segment, scores uniform in
    [0, 1), key lengths 1-3.  Each call is timed cold (L2 flushed before each
    of its replays); one JSON line per buffer length."""
    import numpy as np
    import torch

    import __graft_entry__
    from paper_2511_01282_gb300 import respec as rs
    __graft_entry__.build()
    V, B = 32000, 4
    p = rs.params()
    rng = np.random.default_rng(args.seed)
    props = torch.cuda.get_device_properties(0)
    l2 = int(getattr(props, "L2_cache_size", 0) or (126 << 20))
    flush_buf = torch.ones(2 * l2 // 4, dtype=torch.int32, device="cuda")
    sink = torch.empty((), dtype=torch.int32, device="cuda")
    stream = torch.cuda.Stream()

    def cold_us(fn, n=10):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            fn(stream)
        torch.cuda.synchronize()
        with torch.cuda.graph(g, stream=stream):
            fn(stream)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
        with torch.cuda.stream(stream):
            for a, b in ev:
                torch.amax(flush_buf, dim=0, out=sink)
                a.record(stream)
                g.replay()
                b.record(stream)
        torch.cuda.synchronize()
        return sum(a.elapsed_time(b) for a, b in ev) / n * 1e3

    for t in [int(x) for x in args.lengths.split(",")]:
        bufs = []
        for _ in range(B):
            out = []
            while len(out) < t:
                n = int(rng.integers(8, 65))
                if out and rng.random() < 0.3:
                    a = int(rng.integers(0, max(1, len(out) - n)))
                    out += out[a:a + n]
                else:
                    out += rng.integers(0, V, n).tolist()
            bufs.append(np.array(out[:t], np.int32))
        tok_off = torch.tensor(np.concatenate([[0], np.cumsum([len(x) for x in bufs])]), dtype=torch.int64,
                               device="cuda")
        tokens = torch.from_numpy(np.concatenate(bufs)).cuda()
        scores = torch.from_numpy(rng.random(tokens.numel()).astype(np.float32)).cuda()
        ks = torch.tensor([1, 2, 3, 2][:B] * (B // 4 + 1), dtype=torch.int32, device="cuda")[:B].contiguous()
        t_total = tokens.numel()
        idx = torch.empty(rs.rs_match_index_bytes(B, V, t_total), dtype=torch.uint8, device="cuda")
        z = lambda *sh: torch.zeros(sh, dtype=torch.int32, device="cuda")  # noqa: E731
        o1 = [z(B), z(B, 1024), z(B, p.top_c), z(B, p.top_c), z(B, p.top_c, p.span_len), z(B), z(B)]
        o2 = [z(B), z(B, 1024), z(B, p.top_c), z(B, p.top_c), z(B, p.top_c, p.span_len), z(B), z(B)]
        scan_us = cold_us(lambda sm: rs.rs_match_scan(tokens, tok_off, B, ks, None, scores, p, 1024, *o1,
                                                      stream=sm))
        build_us = cold_us(lambda sm: rs.rs_match_index_build(tokens, tok_off, B, V, t_total, idx, stream=sm), n=3)
        idx_us = cold_us(lambda sm: rs.rs_match_scan_indexed(tokens, tok_off, B, ks, None, scores, p, 1024,
                                                             *o2, V, t_total, idx, stream=sm))
        same = all(bool((a == b).all()) for a, b in zip(o1, o2))
        # one decoding step's update: 8 committed tokens per request join the
        # index (each timed replay appends the same 8 positions again: the
        # index is rebuilt on the shorter buffers before every replay)
        grown = [np.concatenate([x, x[-8:]]) for x in bufs]
        g_off = torch.tensor(np.concatenate([[0], np.cumsum([len(x) for x in grown])]), dtype=torch.int64,
                             device="cuda")
        g_tok = torch.from_numpy(np.concatenate(grown)).cuda()
        st_app = torch.zeros(B, dtype=torch.int32, device="cuda")
        app_us = []
        for _ in range(5):  # eager: the flush keeps the GPU busy while the append is enqueued
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                rs.rs_match_index_build(tokens, tok_off, B, V, t_total, idx, stream=stream)
                torch.amax(flush_buf, dim=0, out=sink)
                a.record(stream)
                rs.rs_match_index_append(g_tok, g_off, B, V, t_total, idx, st_app, stream=stream)
                b.record(stream)
            torch.cuda.synchronize()
            app_us.append(a.elapsed_time(b) * 1e3)
        print(json.dumps(dict(leg="retrieval", B=B, t=t, V=V, scan_us=round(scan_us, 2),
                              indexed_us=round(idx_us, 2), build_us=round(build_us, 1),
                              append8_us=round(sorted(app_us)[2], 2), count=o1[0].tolist(),
                              same_outputs=same, timing="cold: L2 flushed before each call")), flush=True)
    return 0


def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        return run_reference(args, rank, world)
    if args.retrieval:
        return 0 if rank != 0 else run_retrieval(args)
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    try:
        return run_ours(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
