"""Benchmark of the verifier data path: verified tokens/s on the full-response
workload (64 requests, response lengths U{32..256}, 8,847 logit rows of
V = 151,936 bf16, 2.69 GB) and achieved HBM bandwidth of the fused kernel.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gb300|reference]

A step is one fused verification of the whole batch (pr_route: row features,
pooling, score, ship rule; one kernel launch) with the logits resident in HBM.
The batch is larger than L2, so no flush is needed between steps.  The K-step
timed loop is repeated until at least 1.5 s of device time is timed, and the
median repeat is reported, so the clock record has many samples.  On one GPU
the line also carries a `configs` object: the tiny (c1), decode-step (c3),
large ragged (c4) and wide-vocabulary (c5) workloads, each generated in full,
resident in HBM, timed the same way and checked against the oracle on sampled
whole requests; and a `noalloc` record (the allocation-free call beside
pr_route).  A value is printed only when its parity sample passes.  Under
torchrun every rank verifies its own batch (weak scaling, no collective on
the data path); rank 0 prints one JSON line.  ``--impl reference`` times the
float64 CPU oracle on the host cores instead (a bounded sample per step).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_28726_gb300 import workloads as W  # noqa: E402

WORKLOAD = "full"
METRIC = "verified tokens/sec at V=151,936 bf16 and achieved HBM GB/s vs peak (1xGB300)"
UNIT = "tokens/s"
KERNEL_FILES = ("pr_device.cuh", "pr_kernels.cuh", "pro_router.cu")
PROFILE = os.path.join(ROOT, "profiles", "verify_rows_ws_bf16_full_response.md")
HBM_NOMINAL_GBS = 8000.0  # GB300 HBM3e nominal bandwidth, reported beside the measured copy peak


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def reduce_max(value: float, world: int, device) -> float:
    """Max over ranks (the slowest rank sets the job time)."""
    if world == 1:
        return value
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def workload_desc(wl) -> str:
    return ("full-response verify: %d requests, T~U{32..256} (%d rows), V=%d %s, "
            "N(0,1)*s, s~U(1,4), spike +U(0,12) on 70%% of rows" % (
                wl.n_req, wl.n_rows, wl.vocab, wl.dtype))


def algorithmic_bytes(wl) -> int:
    """Bytes one fused launch must move: each row's logits, its token id and
    its 36-byte record (8 floats + flags) written and read back once by the
    pooling epilogue; per request two offsets, 11 aggregates, score, ship and
    flags."""
    per_row = wl.vocab * wl.elem_bytes + 4 + 36 + 36
    per_req = 16 + 44 + 4 + 1 + 4
    return wl.n_rows * per_row + wl.n_req * per_req


def source_sha(files) -> str:
    """Hash of the code of the given csrc files with comments and white space
    left out: it identifies the compiled kernels, so a profile's counters stay
    valid across comment edits and go stale with any change to the code."""
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2608_28726_gb300", "csrc", f)) as fh:
            text = fh.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(" ".join(text.split()).encode())
        h.update(b"\0")
    return h.hexdigest()[:16]


def profiled_file_traffic(path, files, key="dram_bytes_per_launch"):
    """DRAM bytes per launch from a committed ncu summary, if its
    `kernel_source_sha` is that of the current code of `files` (else None)."""
    try:
        text = open(path).read()
    except OSError:
        return None
    vals = {}
    for line in text.splitlines():
        if ":" in line and line.strip().startswith("- "):
            k, v = line.strip()[2:].split(":", 1)
            vals[k.strip()] = v.strip().strip("`")
    if vals.get("kernel_source_sha") != source_sha(files):
        return None
    try:
        return int(vals[key])
    except (KeyError, ValueError):
        return None


def profiled_traffic():
    """The verifier kernel's DRAM bytes per launch on the full-response batch."""
    return profiled_file_traffic(PROFILE, KERNEL_FILES, key="dram_bytes_per_full_launch")


class ClockSampler:
    """nvidia-smi clocks / throttle reasons every 100 ms while the bench runs."""

    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.samples = []
        self.proc = None
        self.index = index
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), [p.strip() for p in line.split(",")]))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)

    def summary(self, t0: float, t1: float):
        inside = [s for (t, s) in self.samples if t0 <= t <= t1]
        window = "timed"
        if len(inside) < 3:
            inside = [s for (_, s) in self.samples]
            window = "whole run (timed region shorter than 3 samples)"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm = [float(s[1]) for s in inside if s[1].replace(".", "").isdigit()]
        mx = [float(s[2]) for s in inside if s[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in inside for i in range(4)
                          if len(s) > 5 + i and s[5 + i].lower().startswith("active")})
        pw = [float(s[3]) for s in inside if s[3].replace(".", "").isdigit()]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "power_w_max": max(pw) if pw else None,
                "reasons": reasons, "samples": len(inside), "window": window}


def oracle_sample(wl, x_host_rows, chosen_host, req_lo: int, req_hi: int, n_threads: int):
    """Oracle on whole requests [req_lo, req_hi) of the workload."""
    import oracle
    off = wl.offsets
    lo, hi = int(off[req_lo]), int(off[req_hi])
    sub_off = off[req_lo:req_hi + 1] - lo
    t0 = time.perf_counter()
    o = oracle.route(x_host_rows, chosen_host, sub_off, wl.w.astype(np.float64), wl.b, wl.tau,
                     n_threads=n_threads)
    dt = time.perf_counter() - t0
    return o, dt, hi - lo


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    wl = W.make(WORKLOAD)
    cores = os.cpu_count() or 1
    # one step = the oracle on one bounded sample of whole requests
    req_hi = 2
    lo, hi = 0, int(wl.offsets[req_hi])
    x, ch = W.rows(wl, lo, hi, device="cpu")
    xs, cs = W.to_oracle_array(x), ch.numpy()
    for _ in range(args.warmup):
        oracle_sample(wl, xs, cs, 0, req_hi, cores)
    times = []
    for _ in range(args.steps):
        _, dt, rows = oracle_sample(wl, xs, cs, 0, req_hi, cores)
        times.append(dt)
    total = sum(times)
    value = (hi - lo) * args.steps / total
    sample = "requests 0..%d of the workload (%d rows of V=%d bf16) per step" % (
        req_hi - 1, hi - lo, wl.vocab)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": workload_desc(wl), "sample_rows_per_step": hi - lo},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ---- timing, parity and the per-configuration records of the verifier ------------------

T_START = time.time()
MIN_TIMED_S = 1.5  # each timed measurement repeats its K-step loop until this much device time
TOL_RTOL, TOL_ATOL, SHIP_BAND = 1e-4, 1e-5, 1e-6  # the verifier's parity bar


def measured_peak():
    peaks_file = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(peaks_file):
        return float(json.load(open(peaks_file))["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def timed_repeats(step, K: int, stream, dev, world: int, B, min_s: float | None = None):
    """Time K back-to-back steps with CUDA events on `stream`, a barrier and a
    synchronize on both sides (max over ranks), and repeat that K-step loop
    until at least `min_s` seconds of device time are timed (at least three
    repeats).  Returns (per-repeat ms per step, wall window, launches in all
    timed repeats)."""
    if min_s is None:
        min_s = MIN_TIMED_S
    per, total_ms = [], 0.0
    launches = 0
    t_wall0 = time.time()
    while len(per) < 3 or total_ms < min_s * 1e3:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier(world)
        torch.cuda.synchronize(dev)
        n0 = B.launch_count()
        e0.record(stream)
        for _ in range(K):
            step()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        barrier(world)
        launches += B.launch_count() - n0
        ms = reduce_max(e0.elapsed_time(e1), world, dev)
        per.append(ms / K)
        total_ms += ms
    return per, (t_wall0, time.time()), launches


def parity_ok(g_agg, g_score, g_ship, g_flags, o, tau):
    """The verifier's parity bar on whole requests: aggregates and scores within
    1e-5 + 1e-4 |oracle|, flags equal, ship equal except where the oracle's
    score is within 1e-6 of tau.  `o` holds the oracle's agg, score, ship and
    req_flags for the same requests, in the same order."""
    ga = np.asarray(g_agg, np.float64)
    gs = np.asarray(g_score, np.float64)
    oa, os_ = np.asarray(o["agg"], np.float64), np.asarray(o["score"], np.float64)

    def close(g, ref):
        nan = np.isnan(g) & np.isnan(ref)
        with np.errstate(invalid="ignore"):
            return bool(np.all(nan | (np.abs(g - ref) <= TOL_ATOL + TOL_RTOL * np.abs(ref))))

    ship_ok = np.all((np.asarray(g_ship) == np.asarray(o["ship"])) |
                     (np.abs(os_ - tau) < SHIP_BAND))
    flags_ok = np.array_equal(np.asarray(g_flags).astype(np.uint32),
                              np.asarray(o["req_flags"]).astype(np.uint32))
    return bool(close(ga, oa) and close(gs, os_) and ship_ok and flags_ok)


def gate_on_parity(rec: dict) -> dict:
    """Verified tokens/s count only for runs whose sampled outputs pass oracle
    parity: a record whose parity failed keeps its timings but no value."""
    if not rec.get("parity", {}).get("ok", False):
        rec["value_withheld"] = "parity with the oracle failed on the sampled requests"
        rec["value"] = None
    return rec


def oracle_on_requests(wl, x_rows_of, reqs, threads: int):
    """The float64 oracle on whole requests `reqs`; x_rows_of(lo, hi) returns
    the device rows [lo, hi) and their token ids.  Returns the oracle's agg,
    score, ship and req_flags stacked in request order, the seconds it took
    and the rows it covered."""
    import oracle
    outs, secs, rows = [], 0.0, 0
    for r in reqs:
        lo, hi = int(wl.offsets[r]), int(wl.offsets[r + 1])
        x, ch = x_rows_of(lo, hi)
        xs, cs = W.to_oracle_array(x), ch.cpu().numpy()
        t0 = time.perf_counter()
        outs.append(oracle.route(xs, cs, np.array([0, hi - lo], np.int64),
                                 wl.w.astype(np.float64), wl.b, wl.tau, n_threads=threads))
        secs += time.perf_counter() - t0
        rows += hi - lo
    stack = {k: np.concatenate([o[k] for o in outs]) for k in ("agg", "score", "ship",
                                                                 "req_flags")}
    return stack, secs, rows


def _route_rec(wl, name, desc, timing, ms, iso_ms, stream_ms, bytes_per_step, rows_per_step,
               world, clocks, launches, K, repeats, parity, graph=None):
    peak, peak_src = measured_peak()
    ach = bytes_per_step / (ms / 1e3) / 1e9
    rec = {
        "workload": desc, "value": rows_per_step * world / (ms / 1e3), "unit": UNIT,
        "ms_per_step": ms, "steps": K, "repeats": repeats, "rows_per_step_per_gpu": rows_per_step,
        "dtype": "f32" if wl.dtype == "f32" else "bf16", "timing": timing,
        "roofline": {"bound": "hbm", "achieved": ach, "peak": peak, "unit": "GB/s",
                     "frac": ach / peak, "traffic": None, "peak_source": peak_src,
                     "kernel": ("verify_rows_ws" if rows_per_step > 1024 else "verify_rows")
                               + "<%s, %s>" % ("f32" if wl.dtype == "f32" else "bf16",
                                               "decode" if name == "decode" else "route"),
                     "algorithmic_bytes_per_step": bytes_per_step,
                     "stream_ms_per_step": stream_ms,
                     "stream_frac": bytes_per_step / (stream_ms / 1e3) / 1e9 / peak,
                     "isolated_ms_per_step": iso_ms,
                     "isolated_frac": bytes_per_step / (iso_ms / 1e3) / 1e9 / peak},
        "clocks": clocks, "gpu_launches": launches, "parity": parity,
        "work_per_row": "Eq. 3 features of the row (Section 3.1), pooled, scored and thresholded "
                        "per request",
    }
    if graph:
        rec["graph"] = graph
    return gate_on_parity(rec)


def measure_route_config(name, B, dev, stream, K, warm, world, sampler, threads, log=None):
    """One of the full-response-style verifier workloads (tiny, ragged, wide),
    resident in HBM; a step is one verification of the whole batch (chunked
    as the workload says).  Returns its record."""
    t_gen = time.time()
    wl = W.make(name)
    copies = 8 if name == "tiny" else 1  # 8 x 45 MB rotated: more than L2 between reuses
    need = copies * wl.n_rows * wl.vocab * wl.elem_bytes
    free, _ = torch.cuda.mem_get_info(dev)
    if need * 1.15 > free:
        raise RuntimeError("%s workload needs %.1f GB, %.1f GB free" % (name, need / 1e9, free / 1e9))
    xs, chs = [], []
    for c in range(copies):
        x = torch.empty(wl.n_rows, wl.vocab, dtype=wl.torch_dtype, device=dev)
        ch = torch.empty(wl.n_rows, dtype=torch.int32, device=dev)
        W.rows(wl, 0, wl.n_rows, device=dev, out=x, chosen_out=ch)
        xs.append(x)
        chs.append(ch)
    torch.cuda.synchronize(dev)
    gen_s = time.time() - t_gen
    off = torch.from_numpy(wl.offsets).to(dev)
    w = torch.from_numpy(wl.w).to(dev)
    ctx = B.pr_ctx_create(dev.index, max_rows=wl.n_rows, max_requests=wl.n_req)
    outs = [(torch.empty(wl.n_req, device=dev), torch.empty(wl.n_req, dtype=torch.uint8, device=dev),
             torch.empty(wl.n_req, dtype=torch.int32, device=dev),
             torch.empty(wl.n_req, 11, device=dev)) for _ in range(copies)]
    chunk = wl.chunk_rows or wl.n_rows
    state = {"c": 0}

    def route_call(c, st):
        for lo in range(0, wl.n_rows, chunk):
            hi = min(wl.n_rows, lo + chunk)
            o = outs[c]
            B.pr_route(ctx, xs[c][lo:hi], chs[c][lo:hi], off, w, wl.b, wl.tau, row_base=lo,
                       score=o[0], ship=o[1], req_flags=o[2], agg=o[3], stream=st)

    def step():
        c = state["c"] % copies
        state["c"] += 1
        route_call(c, stream)

    def timed(overlap):
        B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, overlap)
        for _ in range(warm):
            step()
        torch.cuda.synchronize(dev)
        # steps per timed loop: K, or fewer for steps of many milliseconds (a
        # loop of about half a second; the loop still repeats until
        # MIN_TIMED_S of device time, at least three times)
        t0 = time.perf_counter()
        step()
        torch.cuda.synchronize(dev)
        k_eff = max(3, min(K, int(0.5 / max(time.perf_counter() - t0, 1e-6))))
        state["k"] = k_eff
        return timed_repeats(step, k_eff, stream, dev, world, B)

    iso, _, _ = timed(0)
    per, win, launches = timed(1)
    stream_ms = statistics.median(per)
    ms, reps, timing, graph = stream_ms, len(per), "stream of back-to-back calls", None
    if name == "tiny":
        # launch-bound: one step per rotated copy captured in a CUDA graph, replayed
        gr = torch.cuda.CUDAGraph()
        n0 = B.launch_count()
        with torch.cuda.graph(gr, capture_error_mode="thread_local"):
            gs = torch.cuda.current_stream(dev)
            for c in range(copies):
                route_call(c, gs)
        nodes = B.launch_count() - n0
        for _ in range(3):
            gr.replay()
        torch.cuda.synchronize(dev)
        reps_per = max(1, -(-1000 // copies))
        per_g, win, launches = timed_repeats(gr.replay, reps_per, torch.cuda.current_stream(dev),
                                             dev, world, B)
        ms = statistics.median(per_g) / copies
        launches = nodes * reps_per * len(per_g)
        reps = len(per_g)
        timing = "CUDA graph replays (%d steps per graph, %d replays per repeat)" % (copies,
                                                                                     reps_per)
        graph = {"steps_per_graph": copies, "kernels_per_graph": nodes,
                 "replays_per_repeat": reps_per}
        del gr
    B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, 0)
    clocks = sampler.summary(*win)
    # parity: the last timed outputs of copy 0 on sampled whole requests
    route_call(0, stream)
    torch.cuda.synchronize(dev)
    if name == "tiny":
        reqs = list(range(wl.n_req))
    elif name == "ragged":
        bounds = np.arange(wl.chunk_rows, wl.n_rows, wl.chunk_rows)
        off_np = wl.offsets
        crossing = [r for r in range(wl.n_req)
                    if np.any((off_np[r] < bounds) & (bounds < off_np[r + 1]))]
        reqs = crossing + [0, 511, 1023]
    else:
        reqs = [0, 1, 2, 200, 305, 400, 510, 511]
    o, secs, rows = oracle_on_requests(wl, lambda lo, hi: (xs[0][lo:hi], chs[0][lo:hi]), reqs,
                                       threads)
    g = [t.cpu().numpy()[reqs] for t in outs[0]]
    ok = parity_ok(g[3], g[0], g[1], g[2], o, wl.tau)
    parity = {"requests_checked": len(reqs), "rows_checked": rows, "ok": ok,
              "oracle_tokens_per_s": rows / secs if secs > 0 else None}
    desc = {"tiny": "tiny full-response verify: 8 requests, T~U{16..64} (%d rows), V=%d fp32 "
                    "2*N(0,1) + one spike U(0,8) per row; 8 rotated resident copies",
            "ragged": "large ragged batch: 1,024 requests, lengths lognormal(ln 128, 0.8) "
                      "clipped to [8,1024] (%d rows), V=%d bf16, 8,192-row chunks per step",
            "wide": "wide vocabulary: 512 requests, T~U{64..512} (%d rows), V=%d fp32 "
                    "2*Student-t(3), exact top-1 ties on 10%% of rows, one launch"}[name] % (
                        wl.n_rows, wl.vocab)
    rec = _route_rec(wl, name, desc, timing, ms, statistics.median(iso), stream_ms,
                     algorithmic_bytes(wl) if name != "tiny" else algorithmic_bytes(wl),
                     wl.n_rows, world, clocks, launches, state["k"], reps, parity, graph)
    rec["generation_s"] = gen_s
    rec["l2"] = ("8 rotated copies (360 MB) larger than L2" if name == "tiny" else
                 "inputs (%.1f GB) larger than L2 (129 MB), no flush" % (need / 1e9))
    B.pr_ctx_destroy(ctx)
    del xs, chs, outs
    torch.cuda.empty_cache()
    return rec


def measure_decode_config(B, dev, stream, K, warm, world, sampler, threads, n_steps: int = 1000):
    """The incremental decode-step workload: 256 live slots for 1,000 steps,
    V = 151,936 bf16, the whole trace resident (77.8 GB); a step is one
    pr_decode_step of 256 rows.  Timed as isolated calls, back-to-back calls
    and (headline) CUDA-graph replays of a context reset plus the whole trace.
    Parity: every sampled request that finishes inside the trace against the
    oracle on its rows."""
    t_gen = time.time()
    tr = W.decode_trace(n_steps=n_steps)
    wl = tr.as_workload()
    S, T = tr.n_slots, tr.n_steps
    x_all = torch.empty(T * S, wl.vocab, dtype=wl.torch_dtype, device=dev)
    ch_all = torch.empty(T * S, dtype=torch.int32, device=dev)
    W.rows(wl, 0, T * S, device=dev, out=x_all, chosen_out=ch_all)
    torch.cuda.synchronize(dev)
    gen_s = time.time() - t_gen
    eos = torch.from_numpy(tr.eos).to(dev)
    slot = torch.arange(S, dtype=torch.int32, device=dev)
    w = torch.from_numpy(tr.w).to(dev)
    ctx = B.pr_ctx_create(dev.index, max_rows=S, max_requests=S)
    outs = (torch.empty(S, device=dev), torch.empty(S, dtype=torch.uint8, device=dev),
            torch.empty(S, dtype=torch.int32, device=dev), torch.empty(S, 11, device=dev))
    state = {"t": 0}

    def decode_call(t, st):
        B.pr_decode_step(ctx, x_all[t * S:(t + 1) * S], slot, ch_all[t * S:(t + 1) * S], eos[t], w,
                         tr.b, tr.tau, *outs[:3], agg_out=outs[3], stream=st)

    def step():
        t = state["t"]
        if t == T:
            B.pr_ctx_reset(ctx, stream=stream)
            t = 0
        decode_call(t, stream)
        state["t"] = t + 1

    def timed(overlap):
        B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, overlap)
        for _ in range(warm):
            step()
        torch.cuda.synchronize(dev)
        return timed_repeats(step, max(K, 100), stream, dev, world, B)

    iso, _, _ = timed(0)
    per, _, _ = timed(1)
    stream_ms = statistics.median(per)
    gr = torch.cuda.CUDAGraph()
    n0 = B.launch_count()
    with torch.cuda.graph(gr, capture_error_mode="thread_local"):
        gs = torch.cuda.current_stream(dev)
        B.pr_ctx_reset(ctx, stream=gs)
        for t in range(T):
            decode_call(t, gs)
    nodes = B.launch_count() - n0
    for _ in range(2):
        gr.replay()
    torch.cuda.synchronize(dev)
    per_g, win, _ = timed_repeats(gr.replay, 1, torch.cuda.current_stream(dev), dev, world, B)
    ms = statistics.median(per_g) / T
    launches = nodes * len(per_g)
    B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, 0)
    clocks = sampler.summary(*win)
    del gr

    # parity: one more pass over the trace, untimed, keeping every finished
    # request's outputs (gathered on the device at its EOS step)
    B.pr_ctx_reset(ctx, stream=stream)
    ends = {}
    keep = []
    for t in range(T):
        decode_call(t, stream)
        done = np.nonzero(tr.eos[t])[0]
        if done.size:
            idx = torch.from_numpy(done.astype(np.int64)).to(dev)
            keep.append((t, done, [o.index_select(0, idx) for o in outs]))
    torch.cuda.synchronize(dev)
    for t, done, vals in keep:
        vals = [v.cpu().numpy() for v in vals]
        for j, s in enumerate(done):
            ends[(int(s), t)] = [v[j] for v in vals]
    finished = [(s, t0, L) for (s, t0, L) in tr.requests if t0 + L <= T]
    sample = finished[:12] + finished[-4:]
    import oracle
    g = {"agg": [], "score": [], "ship": [], "req_flags": []}
    o_all = {"agg": [], "score": [], "ship": [], "req_flags": []}
    secs, rows = 0.0, 0
    for (s, t0, L) in sample:
        idx = torch.tensor([(t0 + i) * S + s for i in range(L)], dtype=torch.int64, device=dev)
        xs = W.to_oracle_array(x_all.index_select(0, idx))
        cs = ch_all.index_select(0, idx).cpu().numpy()
        c0 = time.perf_counter()
        o = oracle.route(xs, cs, np.array([0, L], np.int64), tr.w.astype(np.float64), tr.b,
                         tr.tau, n_threads=threads)
        secs += time.perf_counter() - c0
        rows += L
        sc, sh, fl, ag = ends[(s, t0 + L - 1)]
        g["score"].append(sc)
        g["ship"].append(sh)
        g["req_flags"].append(fl)
        g["agg"].append(ag)
        for k in o_all:
            o_all[k].append(o[k][0])
    ok = parity_ok(np.array(g["agg"]), np.array(g["score"]), np.array(g["ship"]),
                   np.array(g["req_flags"]), {k: np.array(v) for k, v in o_all.items()}, tr.tau)
    parity = {"requests_checked": len(sample), "rows_checked": rows, "ok": ok,
              "oracle_tokens_per_s": rows / secs if secs > 0 else None}
    bytes_per_step = S * (wl.vocab * 2 + 4 + 4 + 1) + S * 4
    desc = ("incremental decode-step verify: 256 live slots x %d steps (%d rows, "
            "%.1f GB resident), V=%d bf16 as the full-response rows, lengths U{64..1000}, "
            "one pr_decode_step of 256 rows per step" % (T, T * S, T * S * wl.vocab * 2 / 1e9,
                                                       wl.vocab))
    rec = _route_rec(wl, "decode", desc, "CUDA graph replays (a context reset and the %d-step trace per "
                     "graph)" % T, ms, statistics.median(iso), stream_ms, bytes_per_step, S,
                     world, clocks, launches, T, len(per_g), parity,
                     {"steps_per_graph": T, "kernels_per_graph": nodes, "replays_per_repeat": 1})
    rec["generation_s"] = gen_s
    rec["l2"] = "a %.1f GB trace: every step reads new rows from DRAM" % (T * S * wl.vocab * 2 / 1e9)
    if T != 1000:
        rec["profiling_case"] = "a %d-step trace instead of the 1,000-step one" % T
    B.pr_ctx_destroy(ctx)
    del x_all, ch_all
    torch.cuda.empty_cache()
    return rec


def measure_noalloc(B, x, ch, wl, dev, stream, K, warm, world, n_req: int = 26):
    """pr_route_noalloc (no context, fixed scratch) beside pr_route on the same
    whole batch: the first `n_req` requests of the full-response workload
    (3,994 rows of V = 151,936 bf16), each call one launch."""
    hi = int(wl.offsets[n_req])
    xs, cs = x[:hi], ch[:hi]
    off = torch.from_numpy(wl.offsets[:n_req + 1].copy()).to(dev)
    w = torch.from_numpy(wl.w).to(dev)
    o_na = (torch.empty(n_req, device=dev), torch.empty(n_req, dtype=torch.uint8, device=dev),
            torch.empty(n_req, dtype=torch.int32, device=dev), torch.empty(n_req, 11, device=dev))
    o_rt = tuple(torch.empty_like(t) for t in o_na)
    ctx = B.pr_ctx_create(dev.index, max_rows=hi, max_requests=n_req)

    def na():
        B.pr_route_noalloc(xs, cs, off, w, wl.b, wl.tau, *o_na[:3], agg=o_na[3], stream=stream)

    def rt():
        B.pr_route(ctx, xs, cs, off, w, wl.b, wl.tau, score=o_rt[0], ship=o_rt[1],
                   req_flags=o_rt[2], agg=o_rt[3], stream=stream)

    res = {}
    for name, fn in (("pr_route_noalloc", na), ("pr_route", rt)):
        for _ in range(warm):
            fn()
        torch.cuda.synchronize(dev)
        per, _, _ = timed_repeats(fn, K, stream, dev, world, B, min_s=0.5)
        res[name] = statistics.median(per)
    torch.cuda.synchronize(dev)
    same = (torch.equal(o_na[1], o_rt[1]) and torch.equal(o_na[2], o_rt[2]) and
            bool(torch.all((o_na[0] - o_rt[0]).abs() <= 1e-5 + 1e-4 * o_rt[0].abs())))
    B.pr_ctx_destroy(ctx)
    abytes = hi * (wl.vocab * 2 + 76) + n_req * 69
    peak, _ = measured_peak()
    return {"workload": "full-response rows 0..%d (%d requests), V=%d bf16, one call" % (
                hi - 1, n_req, wl.vocab),
            "ms_per_call": res["pr_route_noalloc"], "pr_route_ms_per_call": res["pr_route"],
            "tokens_per_s": hi / (res["pr_route_noalloc"] / 1e3),
            "frac": abytes / (res["pr_route_noalloc"] / 1e3) / 1e9 / peak,
            "pr_route_frac": abytes / (res["pr_route"] / 1e3) / 1e9 / peak,
            "same_decisions_as_pr_route": bool(same)}


CONFIG_NAMES = {"c1": "tiny", "c3": "decode", "c4": "ragged", "c5": "wide"}


def progress(msg: str):
    """A progress line on stderr with the seconds since the bench started."""
    print("[bench %.1f s] %s" % (time.time() - T_START, msg), file=sys.stderr, flush=True)


def run_gb300(args):
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2608_28726_gb300 import build as prbuild
    prbuild.build()
    from paper_2608_28726_gb300 import binding as B

    wl = W.make(WORKLOAD, n_req=args.requests or None)
    x, ch = W.rows(wl, 0, wl.n_rows, device=dev)
    off = torch.from_numpy(wl.offsets).to(dev)
    w = torch.from_numpy(wl.w).to(dev)
    ctx = B.pr_ctx_create(local, max_rows=wl.n_rows, max_requests=wl.n_req)
    stream = torch.cuda.current_stream(dev)
    score = torch.empty(wl.n_req, device=dev)
    ship = torch.empty(wl.n_req, dtype=torch.uint8, device=dev)
    rflags = torch.empty(wl.n_req, dtype=torch.int32, device=dev)
    agg = torch.empty(wl.n_req, 11, device=dev)

    def step():
        B.pr_route(ctx, x, ch, off, w, wl.b, wl.tau, score=score, ship=ship, req_flags=rflags,
                   agg=agg, stream=stream)

    sampler = ClockSampler(local)
    sampler.start()
    K = args.steps
    warm = max(3, args.warmup)
    min_s = min(0.05, MIN_TIMED_S) if args.skip_host else MIN_TIMED_S

    progress("headline workload generated")
    # (1) isolated launches: one launch at a time (no overlap between steps)
    B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, 0)
    for _ in range(warm):
        step()
    torch.cuda.synchronize(dev)
    iso_per, _, _ = timed_repeats(step, K, stream, dev, world, B, min_s=min_s)
    isolated_ms = statistics.median(iso_per)

    # (2) the headline: K back-to-back steps, each allowed to start while the
    # previous one finishes (programmatic dependent launch; results identical),
    # the K-step loop repeated until enough time is timed; median over repeats
    B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, 1)
    for _ in range(warm):
        step()
    torch.cuda.synchronize(dev)
    per, (t_wall0, t_wall1), launches = timed_repeats(step, K, stream, dev, world, B, min_s=min_s)
    ms_step = statistics.median(per)
    B.pr_ctx_set_option(ctx, B.PR_OPT_OVERLAP, 0)
    clocks = sampler.summary(t_wall0, t_wall1)
    if args.skip_host:
        sampler.stop()
        if rank == 0:
            print(json.dumps({"profiling_case": True, "rows": wl.n_rows, "steps": K,
                              "ms_per_step": ms_step, "gpu_launches": launches}))
        B.pr_ctx_destroy(ctx)
        return 0

    progress("headline timed")
    # end to end from pinned host memory through the public C ABI (without
    # the clock sampler's nvidia-smi process beside it)
    sampler.stop()
    hx = x.cpu().pin_memory()
    hc = ch.cpu().pin_memory()
    hoff = torch.from_numpy(wl.offsets).pin_memory()
    hw = torch.from_numpy(wl.w).pin_memory()
    hs = torch.empty(wl.n_req).pin_memory()
    hsh = torch.empty(wl.n_req, dtype=torch.uint8).pin_memory()
    hf = torch.empty(wl.n_req, dtype=torch.int32).pin_memory()
    ctx_h = B.pr_ctx_create(local, max_rows=wl.n_rows, max_requests=wl.n_req)
    e2e_steps = max(3, min(K, 10))

    def e2e_step():
        B.pr_route_host(ctx_h, hx, hc, hoff, hw, wl.b, wl.tau, chunk_rows=512, score=hs, ship=hsh,
                        req_flags=hf, stream=stream)

    e2e_step()
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    barrier(world)
    e2e_s = reduce_max(time.perf_counter() - t0, world, dev)
    B.pr_ctx_destroy(ctx_h)
    del hx, hc
    sampler.start()

    h2d = wl.n_rows * wl.vocab * 2 + hc_bytes(wl)
    d2h = wl.n_req * (4 + 1 + 4)
    rows_all = wl.n_rows * world
    value = rows_all / (ms_step / 1e3)
    e2e_value = rows_all * e2e_steps / e2e_s

    abytes = algorithmic_bytes(wl)
    achieved = abytes / (ms_step / 1e3) / 1e9
    isolated_achieved = abytes / (isolated_ms / 1e3) / 1e9
    peak, peak_src = measured_peak()
    cores = os.cpu_count() or 1

    progress("end to end timed")
    line = None
    configs = {}
    noalloc = None
    if rank == 0:
        # parity of the timed run's outputs on a sample of whole requests, and
        # the oracle's own speed on that sample (the CPU baseline)
        import oracle
        oracle.build()
        req_hi = 8
        lo, hi = 0, int(wl.offsets[req_hi])
        xs = W.to_oracle_array(x[lo:hi])
        cs = ch[lo:hi].cpu().numpy()
        o, dt, rows = oracle_sample(wl, xs, cs, 0, req_hi, cores)
        # the same oracle on one core, on request 0 alone
        hi1 = int(wl.offsets[1])
        _, dt1, rows1 = oracle_sample(wl, xs[:hi1], cs[:hi1], 0, 1, 1)
        ok = (parity_ok(agg[:req_hi].cpu().numpy(), score[:req_hi].cpu().numpy(),
                        ship[:req_hi].cpu().numpy(), rflags[:req_hi].cpu().numpy(), o, wl.tau)
              and bool(np.all(hsh[:req_hi].numpy() == ship[:req_hi].cpu().numpy())))
        if not args.requests:
            noalloc = measure_noalloc(B, x, ch, wl, dev, stream, K, warm, world)
    B.pr_ctx_destroy(ctx)
    del x, ch
    torch.cuda.empty_cache()
    progress("headline parity, CPU baseline and pr_route_noalloc done")

    if rank == 0 and world == 1 and args.configs != "none":
        for key in [k.strip() for k in args.configs.split(",") if k.strip()]:
            name = CONFIG_NAMES[key]
            try:
                if name == "decode":
                    configs[key] = measure_decode_config(B, dev, stream, K, warm, world, sampler,
                                                         cores)
                else:
                    configs[key] = measure_route_config(name, B, dev, stream, K, warm, world,
                                                        sampler, cores)
            except (RuntimeError, torch.cuda.OutOfMemoryError) as e:
                torch.cuda.empty_cache()
                configs[key] = {"workload": name, "value": None, "error": str(e).splitlines()[0]}
            progress("config %s (%s) done" % (key, name))
    sampler.stop()

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": warm, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": workload_desc(wl), "rows_per_step_per_gpu": wl.n_rows,
                       "logit_bytes_per_step_per_gpu": wl.n_rows * wl.vocab * 2,
                       "l2": "inputs (2.69 GB) larger than L2 (129 MB), no flush",
                       "overlap": "back-to-back steps may overlap (PR_OPT_OVERLAP: programmatic "
                                  "dependent launch); isolated launches reported in roofline",
                       "timing": "the K-step loop repeated %d times (at least %.1f s of device "
                                 "time); ms_per_step is the median repeat" % (len(per), min_s),
                       "parallelism": "dp%d (independent batches)" % world},
            "repeats": len(per),
            "ms_per_step_repeats": {"min": min(per), "median": ms_step, "max": max(per)},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": profiled_traffic(),
                         "kernel": "verify_rows_ws<bf16, route>", "peak_source": peak_src,
                         "algorithmic_bytes_per_launch": abytes,
                         "avg_launch_ms": ms_step,
                         "isolated_launch_ms": isolated_ms,
                         "isolated_achieved": isolated_achieved,
                         "isolated_frac": isolated_achieved / peak,
                         "nominal_peak": HBM_NOMINAL_GBS,
                         "frac_of_nominal": achieved / HBM_NOMINAL_GBS},
            "cpu_baseline": {"value": rows / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": "requests 0..%d (%d rows), float64 C oracle, %d threads" % (
                                 req_hi - 1, rows, cores)},
            "cpu_baseline_one_core": {"value": rows1 / dt1, "unit": UNIT, "cores": 1,
                                      "kind": "oracle",
                                      "sample": "request 0 (%d rows), float64 C oracle, 1 thread"
                                                % rows1},
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d * world,
                    "d2h_bytes_per_step": d2h, "api": "pr_route_host (pinned host buffers)"},
            "gpu_launches": launches,
            "timed_steps_total": K * len(per),
            "clocks": clocks,
            "parity": {"requests_checked": req_hi, "rows_checked": rows, "ok": ok},
        }
        if configs:
            line["configs"] = configs
        if noalloc:
            line["noalloc"] = noalloc
        line = gate_on_parity(line)
        if line["value"] is None:
            line["e2e"]["value"] = None
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def hc_bytes(wl) -> int:
    """Host-to-device bytes of one end-to-end step beside the logits: token
    ids, offsets and scorer weights."""
    return wl.n_rows * 4 + (wl.n_req + 1) * 8 + 11 * 4


def run_other_workload(args):
    """One of the four other verifier workloads on its own line, measured as
    the default run's `configs` records are."""
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2608_28726_gb300 import build as prbuild
    prbuild.build()
    from paper_2608_28726_gb300 import binding as B
    stream = torch.cuda.current_stream(dev)
    sampler = ClockSampler(local)
    sampler.start()
    warm = max(3, args.warmup)
    cores = os.cpu_count() or 1
    if args.workload == "decode":
        rec = measure_decode_config(B, dev, stream, args.steps, warm, world, sampler, cores,
                                    n_steps=args.decode_steps)
    else:
        rec = measure_route_config(args.workload, B, dev, stream, args.steps, warm, world,
                                   sampler, cores)
    sampler.stop()
    if rank == 0:
        line = {"metric": "verified tokens/sec (%s workload)" % args.workload,
                "value": rec["value"], "unit": UNIT, "n_gpus": world, "steps": rec["steps"],
                "warmup": warm, "ms_per_step": rec["ms_per_step"], "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": rec["dtype"],
                "data": "synthetic",
                "config": {"workload": rec["workload"], "timing": rec["timing"],
                           "rows_per_step_per_gpu": rec["rows_per_step_per_gpu"],
                           "l2": rec["l2"]},
                "roofline": rec["roofline"], "gpu_launches": rec["gpu_launches"],
                "clocks": rec["clocks"], "parity": rec["parity"]}
        if "graph" in rec:
            line["graph"] = rec["graph"]
        if "value_withheld" in rec:
            line["value_withheld"] = rec["value_withheld"]
        if "profiling_case" in rec:
            line["profiling_case"] = rec["profiling_case"]
        print(json.dumps(line))
    return 0


HEAD_FILES = ("pr_device.cuh", "pr_head.cuh", "pr_head_api.cu")
HEAD_PROFILE = os.path.join(ROOT, "profiles", "head_attn_f32_full_response.md")
# fp32 CUDA-core peak: 152 SMs x 128 FMA lanes x 2 flop x 2,070 MHz (maximum SM clock)
FP32_PEAK_TFLOPS = 152 * 128 * 2 * 2.070e9 / 1e12
# dense TF32 tensor rate against dense bf16, nominal (1.1 / 2.25 PFLOP/s)
TF32_PER_BF16 = 1.1 / 2.25


def tf32_peak():
    """(TF/s, source): the measured bf16 burst rate x the nominal TF32 ratio."""
    peaks_file = os.path.join(ROOT, "MEASURED_PEAKS.json")
    peaks = json.load(open(peaks_file)) if os.path.exists(peaks_file) else {}
    bf16 = float(peaks.get("bf16_tflops", 0.0) or 0.0)
    if bf16 > 0:
        return bf16 * TF32_PER_BF16, "measured bf16 burst (%.1f TF/s) x 1.1/2.25" % bf16
    return 1900.0 * TF32_PER_BF16, "fallback bf16 1,900 TF/s x 1.1/2.25"


def head_flops(lengths, n_layers: int):
    """Algorithmic flops of the scorer head: per layer and token the QKV,
    output, and two feed-forward projections (2 x 64 x (192 + 64 + 128 + 128)),
    per layer, request and head the scores and the weighted values
    (2 x 2 x 16 x T^2, four heads); the embedding and pooling are left out.
    Returns (whole step, one attention launch)."""
    T = np.asarray(lengths, np.float64)
    attn = float(4 * 2 * 2 * 16 * np.sum(T * T))
    rows = float(2 * 64 * (3 * 64 + 64 + 2 * 128) * np.sum(T))
    return n_layers * (rows + attn), attn


def head_oracle_sample(req_hi: int, n_layers: int):
    """The float64 head oracle on requests 0 .. req_hi - 1 of the head workload,
    in a child process with one BLAS / OpenMP thread.  Returns (seconds,
    scores, ship)."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    out = subprocess.run([sys.executable, os.path.abspath(__file__), "--head-oracle-sample",
                          str(req_hi), "--head-layers", str(n_layers)],
                         env=env, capture_output=True, text=True, check=True)
    d = json.loads(out.stdout.strip().splitlines()[-1])
    return d["seconds"], np.asarray(d["score"], np.float64), np.asarray(d["ship"], np.uint8)


def head_oracle_child(req_hi: int, n_layers: int):
    from oracle import head as ohead
    wl = W.make(WORKLOAD)
    feat_h, offsets = W.head_features(wl.lengths, seed=4001)
    w_h = W.head_weights(n_layers)
    hi = int(offsets[req_hi])
    t0 = time.perf_counter()
    so, po, _ = ohead.head_score(feat_h[:hi].astype(np.float64), np.zeros(hi, np.uint32),
                                 offsets[:req_hi + 1], w_h.astype(np.float64), n_layers, wl.tau)
    dt = time.perf_counter() - t0
    print(json.dumps({"seconds": dt, "score": so.tolist(), "ship": po.tolist()}))
    return 0


def run_head_workload(args):
    """The transformer scorer head (2 layers) on the full-response request
    layout: 64 requests, T ~ U{32..256}, seeded feature records resident in HBM;
    the activations fit in L2, so L2 is flushed between timed steps."""
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2608_28726_gb300 import build as prbuild
    prbuild.build()
    from paper_2608_28726_gb300 import binding as B
    n_layers = 2
    wl = W.make(WORKLOAD)
    lengths = wl.lengths
    feat_h, offsets = W.head_features(lengths, seed=4001)
    w_h = W.head_weights(n_layers)
    feat = torch.from_numpy(feat_h).to(dev)
    off = torch.from_numpy(offsets).to(dev)
    w = torch.from_numpy(w_h).to(dev)
    n_req, n_rows = len(lengths), int(offsets[-1])
    ctx = B.pr_ctx_create(local, max_rows=0, max_requests=1)
    stream = torch.cuda.current_stream(dev)
    score = torch.empty(n_req, device=dev)
    ship = torch.empty(n_req, dtype=torch.uint8, device=dev)
    rflags = torch.empty(n_req, dtype=torch.int32, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # 256 MB > L2

    def step():
        B.pr_head_score(ctx, feat, off, w, n_layers, wl.tau, score=score, ship=ship,
                        req_flags=rflags, stream=stream)

    K = args.steps
    sampler = ClockSampler(local)
    sampler.start()

    def timed(timing: int):
        B.pr_ctx_set_option(ctx, B.PR_OPT_TIMING, timing)
        for _ in range(max(3, args.warmup)):
            step()
        torch.cuda.synchronize(dev)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(K)]
        kernel_ms = []
        barrier(world)
        torch.cuda.synchronize(dev)
        n0 = B.launch_count()
        for i in range(K):
            flush.zero_()
            ev[i][0].record(stream)
            step()
            ev[i][1].record(stream)
            if timing:
                kernel_ms.append(B.pr_ctx_kernel_times(ctx))
        torch.cuda.synchronize(dev)
        barrier(world)
        total = sum(a.elapsed_time(b) for a, b in ev)
        return reduce_max(total, world, dev) / K, B.launch_count() - n0, kernel_ms

    # the K-step loop repeated until MIN_TIMED_S of wall time (at least three
    # times), so that the clock record covers a window of many samples; the
    # median repeat is the step time
    t_wall0 = time.time()
    reps, launches = [], 0
    while len(reps) < 3 or time.time() - t_wall0 < MIN_TIMED_S:
        ms_r, n_r, _ = timed(0)
        reps.append(ms_r)
        launches += n_r
    ms = statistics.median(reps)
    t_wall1 = time.time()
    iso_ms, _, kernel_ms = timed(1)
    B.pr_ctx_set_option(ctx, B.PR_OPT_TIMING, 0)
    clocks = sampler.summary(t_wall0, t_wall1)
    sampler.stop()
    attn_idx = [2 + 2 * l for l in range(n_layers)]
    attn_ms = float(np.mean([k[i] for k in kernel_ms for i in attn_idx]))
    per_kernel = np.mean(np.asarray(kernel_ms), axis=0).tolist()

    # end to end through the public API: features and offsets from pinned host
    # memory, scores, ship bits and flags back to pinned host memory
    hf, ho = torch.from_numpy(feat_h).pin_memory(), torch.from_numpy(offsets).pin_memory()
    hs = torch.empty(n_req).pin_memory()
    hsh = torch.empty(n_req, dtype=torch.uint8).pin_memory()
    hfl = torch.empty(n_req, dtype=torch.int32).pin_memory()
    dfeat, doff = torch.empty_like(feat), torch.empty_like(off)

    def e2e_step():
        dfeat.copy_(hf, non_blocking=True)
        doff.copy_(ho, non_blocking=True)
        B.pr_head_score(ctx, dfeat, doff, w, n_layers, wl.tau, score=score, ship=ship,
                        req_flags=rflags, stream=stream)
        hs.copy_(score, non_blocking=True)
        hsh.copy_(ship, non_blocking=True)
        hfl.copy_(rflags, non_blocking=True)
        torch.cuda.synchronize(dev)

    e2e_step()
    e2e_steps = max(3, min(K, 50))
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    barrier(world)
    e2e_s = reduce_max(time.perf_counter() - t0, world, dev)
    h2d = hf.numel() * 4 + ho.numel() * 8
    d2h = n_req * (4 + 1 + 4)

    step_flops, attn_flops = head_flops(lengths, n_layers)
    achieved = attn_flops / (attn_ms / 1e3) / 1e12
    tf32_pk, tf32_src = tf32_peak()
    if rank == 0:
        req_hi = n_req  # the whole workload: under a second of oracle time
        lo, hi = 0, int(offsets[req_hi])
        dt, so, po = head_oracle_sample(req_hi, n_layers)
        cores = 1
        g = score[:req_hi].cpu().numpy().astype(np.float64)
        ok = bool(np.all(np.abs(g - so) <= 1e-5) and
                  np.all((ship[:req_hi].cpu().numpy() == po) | (np.abs(so - wl.tau) < 1e-6)))
        print(json.dumps({
            "metric": "scored tokens/sec (transformer scorer head, %d layers, 64-request "
                      "full-response layout)" % n_layers,
            "value": n_rows * world / (ms / 1e3), "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": "scorer head: %d requests, T~U{32..256} (%d rows), seeded "
                                   "feature records, seeded weights (67,329 floats)" % (
                                       n_req, n_rows),
                       "l2": "256 MB written between timed steps (flush)",
                       "n_layers": n_layers,
                       "timing": "the K-step loop repeated %d times (at least %.1f s); "
                                 "ms_per_step is the median repeat" % (len(reps), MIN_TIMED_S)},
            "repeats": len(reps),
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": tf32_pk,
                         "unit": "TFLOP/s", "frac": achieved / tf32_pk,
                         "traffic": profiled_file_traffic(HEAD_PROFILE, HEAD_FILES),
                         "kernel": "head_attn",
                         "peak_source": tf32_src + "; the contractions run as three TF32 "
                                        "products per fp32 product",
                         "fp32_cuda_core_frac": achieved / FP32_PEAK_TFLOPS,
                         "algorithmic_flops_per_launch": attn_flops,
                         "avg_launch_ms": attn_ms,
                         "step_flops": step_flops,
                         "step_tflops": step_flops / (ms / 1e3) / 1e12,
                         "isolated_kernel_ms": per_kernel,
                         "isolated_step_ms": iso_ms},
            "cpu_baseline": {"value": (hi - lo) / dt, "unit": UNIT, "cores": cores,
                             "kind": "oracle",
                             "sample": "requests 0..%d (%d rows), float64 numpy head oracle" % (
                                 req_hi - 1, hi - lo)},
            "e2e": {"value": n_rows * world * e2e_steps / e2e_s, "unit": UNIT,
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "api": "pr_head_score with host copies of features, offsets and results"},
            "gpu_launches": launches,
            "clocks": clocks,
            "parity": {"requests_checked": req_hi, "ok": ok},
        }))
    B.pr_ctx_destroy(ctx)
    return 0


LM_FILES = ("pr_device.cuh", "pr_kernels.cuh", "pr_lmhead.cuh", "pr_lmhead_api.cu")
LM_PROFILE = os.path.join(ROOT, "profiles", "lm_fused_bf16_full_response.md")
LM_D = 3584


def lm_oracle_child(n_sample: int):
    """The float64 oracle on the first n_sample rows of the LM-head workload
    (inputs regenerated on the CPU from the same seeds)."""
    from oracle import lmhead
    wl = W.make(WORKLOAD)
    hidden, weight, chosen = W.lmhead_inputs(wl.n_rows, LM_D, wl.vocab, device="cpu")
    hb = hidden[:n_sample].contiguous().view(torch.int16).numpy().view(np.uint16)
    wb = weight.contiguous().view(torch.int16).numpy().view(np.uint16)
    t0 = time.perf_counter()
    o = lmhead.features(hb, wb, chosen[:n_sample].numpy(), K=20,
                        offsets=np.array([0, n_sample], np.int64))
    dt = time.perf_counter() - t0
    print(json.dumps({"seconds": dt, "feat": o["feat"].tolist()}))
    return 0


def run_lmhead_workload(args):
    """The LM head fused with the row reduction on the full-response batch:
    8,847 hidden states of d = 3,584 against a 151,936 x 3,584 bf16 head."""
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2608_28726_gb300 import build as prbuild
    prbuild.build()
    from paper_2608_28726_gb300 import binding as B
    wl = W.make(WORKLOAD)
    n, V, d = wl.n_rows, wl.vocab, LM_D
    # generated on the CPU (the oracle's child process draws the same values)
    hidden, weight, chosen = (t.to(dev) for t in W.lmhead_inputs(n, d, V, device="cpu"))
    off = torch.from_numpy(wl.offsets).to(dev)
    if args.lm_rows > 0:  # the first rows only, as one request (e.g. one decode step's batch)
        n = min(args.lm_rows, n)
        hidden, chosen = hidden[:n].contiguous(), chosen[:n].contiguous()
        off = torch.tensor([0, n], dtype=torch.int64, device=dev)
    ctx = B.pr_ctx_create(local, max_rows=n, max_requests=wl.n_req)
    stream = torch.cuda.current_stream(dev)
    feat = torch.empty(n, 8, device=dev)
    top2 = torch.empty(n, 2, dtype=torch.int32, device=dev)
    rf = torch.empty(n, dtype=torch.int32, device=dev)

    def step():
        B.pr_lmhead_features(ctx, hidden, weight, chosen, 20, offsets=off, feat=feat, top2=top2,
                             row_flags=rf, stream=stream)

    K = args.steps
    sampler = ClockSampler(local)
    sampler.start()
    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize(dev)
    n0 = B.launch_count()
    t_wall0 = time.time()
    e0.record(stream)
    for _ in range(K):
        step()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    t_wall1 = time.time()
    barrier(world)
    launches = B.launch_count() - n0
    ms = reduce_max(e0.elapsed_time(e1), world, dev) / K
    clocks = sampler.summary(t_wall0, t_wall1)
    # per kernel (PR_OPT_TIMING)
    B.pr_ctx_set_option(ctx, B.PR_OPT_TIMING, 1)
    kms = []
    for _ in range(max(3, min(K, 10))):
        step()
        kms.append(B.pr_ctx_kernel_times(ctx))
    B.pr_ctx_set_option(ctx, B.PR_OPT_TIMING, 0)
    fused_ms, merge_ms = [float(x) for x in np.mean(np.asarray(kms), axis=0)]
    flags = B.pr_ctx_flags(ctx, clear=True)
    # the unfused path for comparison: cuBLAS writes the bf16 logits, then the
    # verifier reads them back (pr_token_features)
    logits = torch.empty(n, V, dtype=torch.bfloat16, device=dev)
    ufeat = torch.empty_like(feat)

    def unfused():
        torch.matmul(hidden, weight.t(), out=logits)
        B.pr_token_features(ctx, logits, chosen, 20, offsets=off, feat=ufeat, stream=stream)

    for _ in range(3):
        unfused()
    torch.cuda.synchronize(dev)
    u0, u1, u2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
    KU = max(3, K)  # the same number of steps as the fused leg (same power-capped regime)
    gemm_ms = feat_ms = 0.0
    for _ in range(KU):
        u0.record(stream)
        torch.matmul(hidden, weight.t(), out=logits)
        u1.record(stream)
        B.pr_token_features(ctx, logits, chosen, 20, offsets=off, feat=ufeat, stream=stream)
        u2.record(stream)
        torch.cuda.synchronize(dev)
        gemm_ms += u0.elapsed_time(u1)
        feat_ms += u1.elapsed_time(u2)
    gemm_ms /= KU
    feat_ms /= KU
    del logits
    sampler.stop()

    # decode steps (with --lm-rows): the n rows as live slots, each step through
    # pr_lmhead_decode_step, against cuBLAS logits + pr_decode_step
    decode = None
    if args.lm_rows > 0:
        dctx = B.pr_ctx_create(local, max_rows=n, max_requests=n)
        slot = torch.arange(n, dtype=torch.int32, device=dev)
        eos0 = torch.zeros(n, dtype=torch.uint8, device=dev)
        dw = torch.from_numpy(wl.w).to(dev)
        dsc = torch.empty(n, device=dev)
        dsh = torch.empty(n, dtype=torch.uint8, device=dev)
        dfl = torch.empty(n, dtype=torch.int32, device=dev)
        dlog = torch.empty(n, V, dtype=torch.bfloat16, device=dev)
        KD = max(3, min(K, 200))

        def dec_fused():
            B.pr_lmhead_decode_step(dctx, hidden, weight, slot, chosen, eos0, dw, wl.b, wl.tau,
                                    dsc, dsh, dfl, stream=stream)

        def dec_unfused():
            torch.matmul(hidden, weight.t(), out=dlog)
            B.pr_decode_step(dctx, dlog, slot, chosen, eos0, dw, wl.b, wl.tau, dsc, dsh, dfl,
                             stream=stream)

        dres = {}
        for name_, fn in (("fused", dec_fused), ("unfused", dec_unfused)):
            B.pr_ctx_reset(dctx, stream=stream)
            for _ in range(3):
                fn()
            torch.cuda.synchronize(dev)
            d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            d0.record(stream)
            for _ in range(KD):
                fn()
            d1.record(stream)
            torch.cuda.synchronize(dev)
            dres[name_] = d0.elapsed_time(d1) / KD
        decode = {"slots": n, "steps": KD, "fused_ms_per_step": dres["fused"],
                  "unfused_ms_per_step": dres["unfused"],
                  "speedup_of_fused": dres["unfused"] / dres["fused"],
                  "api": "pr_lmhead_decode_step vs cuBLAS logits + pr_decode_step"}
        del dlog
        B.pr_ctx_destroy(dctx)

    # e2e: the step's hidden states from pinned host memory, its records back
    hh = hidden.cpu().pin_memory()
    hfeat = torch.empty(n, 8).pin_memory()
    dh = torch.empty_like(hidden)

    def e2e_step():
        dh.copy_(hh, non_blocking=True)
        B.pr_lmhead_features(ctx, dh, weight, chosen, 20, offsets=off, feat=feat, top2=top2,
                             row_flags=rf, stream=stream)
        hfeat.copy_(feat, non_blocking=True)
        torch.cuda.synchronize(dev)

    e2e_step()
    e2e_steps = max(3, min(K, 10))
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    barrier(world)
    e2e_s = reduce_max(time.perf_counter() - t0, world, dev)

    flops = 2.0 * n * d * V
    peaks_file = os.path.join(ROOT, "MEASURED_PEAKS.json")
    peaks = json.load(open(peaks_file)) if os.path.exists(peaks_file) else {}
    peak = float(peaks.get("bf16_tflops_sustained", 1700.0))
    achieved = flops / (fused_ms / 1e3) / 1e12
    if rank == 0:
        n_sample = 4
        out = subprocess.run([sys.executable, os.path.abspath(__file__), "--lm-oracle-child",
                              str(n_sample)],
                             env=dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1",
                                      MKL_NUM_THREADS="1"),
                             capture_output=True, text=True, check=True)
        dd = json.loads(out.stdout.strip().splitlines()[-1])
        fo = np.asarray(dd["feat"], np.float64)
        fg = feat[:n_sample].cpu().numpy().astype(np.float64)
        fg[:, 5] = fo[:, 5]  # rho: the sample is one request of n_sample rows on the oracle side
        ok = bool(np.all(np.abs(fg - fo) <= 1e-4 + 1e-4 * np.abs(fo))) and flags == 0
        print(json.dumps({
            "metric": "verified tokens/sec with the LM head fused (logits never written), "
                      "V=151,936, d=3,584",
            "value": n * world / (ms / 1e3), "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": "LM head + row features: %d hidden states (%s), d=%d, V=%d "
                                   "bf16 head (1.09 GB), seeded" % (
                                       n, "the full-response layout" if args.lm_rows <= 0
                                       else "the first rows of the full-response batch, one "
                                            "request", d, V),
                       "l2": "inputs (1.15 GB) larger than L2 (129 MB), no flush"},
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak,
                         "unit": "TFLOP/s", "frac": achieved / peak,
                         "traffic": profiled_file_traffic(LM_PROFILE, LM_FILES),
                         "kernel": "lm_fused (tcgen05)",
                         "peak_source": "measured cuBLAS bf16, sustained (%.1f burst)" %
                                        float(peaks.get("bf16_tflops", 0.0)),
                         "algorithmic_flops_per_launch": flops, "avg_launch_ms": fused_ms,
                         "merge_ms": merge_ms},
            "unfused": {"cublas_gemm_ms": gemm_ms, "pr_token_features_ms": feat_ms,
                        "ms_per_step": gemm_ms + feat_ms,
                        "logit_bytes_written_and_read": n * V * 2,
                        "speedup_of_fused": (gemm_ms + feat_ms) / ms},
            "decode_steps": decode,
            "cpu_baseline": {"value": n_sample / dd["seconds"], "unit": UNIT, "cores": 1,
                             "kind": "oracle",
                             "sample": "rows 0..%d: float64 product and features" % (n_sample - 1)},
            "e2e": {"value": n * world * e2e_steps / e2e_s, "unit": UNIT,
                    "h2d_bytes_per_step": n * d * 2, "d2h_bytes_per_step": n * 32,
                    "api": "pr_lmhead_features after a host copy of the hidden states "
                           "(the head's weights resident)"},
            "gpu_launches": launches,
            "clocks": clocks,
            "parity": {"rows_checked": n_sample, "ok": ok, "flags": flags},
        }))
    B.pr_ctx_destroy(ctx)
    return 0


QNT_FILES = ("pr_device.cuh", "pr_quant.cuh", "pr_quant_api.cu")
QNT_PROFILE = os.path.join(ROOT, "profiles", "qmlp_requests_f32_ragged.md")
# shared-memory bandwidth: 152 SMs x 32 banks x 4 bytes x 2,070 MHz


def qnt_bytes(n_rows: int, n_req: int) -> int:
    """Algorithmic DRAM bytes of one quantile-scorer launch: each row's 32-byte
    feature record read once, the offsets, the MLP's 6,081 weights, and per
    request a score, a ship byte and a flag word written."""
    return 32 * n_rows + 8 * (n_req + 1) + 4 * 6081 + 9 * n_req


Q_LAYOUTS = {"ragged": "ragged", "full": "full"}  # request layout -> workload it is taken from


def qnt_oracle_child(layout: str = "ragged"):
    from oracle import quantile as oq
    wl = W.make(Q_LAYOUTS[layout])
    feat, offsets = W.head_features(wl.lengths, seed=4001)
    w = W.qmlp_weights()
    t0 = time.perf_counter()
    so, po, fo, mo = oq.quantile_score(feat.astype(np.float64), np.zeros(int(offsets[-1]), np.uint32),
                                       offsets, w.astype(np.float64), wl.tau)
    dt = time.perf_counter() - t0
    print(json.dumps({"seconds": dt, "score": so.tolist(), "ship": po.tolist()}))
    return 0


def run_quantile_workload(args):
    """The quantile-summary + MLP aggregator on the ragged request layout
    (1,024 requests, lognormal lengths, 181,659 rows) or, with --q-layout
    full, the full-response layout (64 requests, T ~ U{32..256}, 8,847 rows)."""
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2608_28726_gb300 import build as prbuild
    prbuild.build()
    from paper_2608_28726_gb300 import binding as B
    wl = W.make(Q_LAYOUTS[args.q_layout])
    feat_h, offsets = W.head_features(wl.lengths, seed=4001)
    w_h = W.qmlp_weights()
    feat, off = torch.from_numpy(feat_h).to(dev), torch.from_numpy(offsets).to(dev)
    w = torch.from_numpy(w_h).to(dev)
    n_req, n_rows = wl.n_req, int(offsets[-1])
    ctx = B.pr_ctx_create(local, max_rows=0, max_requests=1)
    stream = torch.cuda.current_stream(dev)
    score = torch.empty(n_req, device=dev)
    ship = torch.empty(n_req, dtype=torch.uint8, device=dev)
    rflags = torch.empty(n_req, dtype=torch.int32, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def step():
        B.pr_quantile_score(ctx, feat, off, w, wl.tau, score=score, ship=ship, req_flags=rflags,
                            want_summary=False, stream=stream)

    K = args.steps
    sampler = ClockSampler(local)
    sampler.start()
    for _ in range(max(3, args.warmup)):
        step()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    barrier(world)
    torch.cuda.synchronize(dev)
    n0 = B.launch_count()
    t_wall0 = time.time()
    for i in range(K):
        flush.zero_()
        ev[i][0].record(stream)
        step()
        ev[i][1].record(stream)
    torch.cuda.synchronize(dev)
    t_wall1 = time.time()
    barrier(world)
    launches = B.launch_count() - n0
    ms = reduce_max(sum(a.elapsed_time(b) for a, b in ev), world, dev) / K
    clocks = sampler.summary(t_wall0, t_wall1)
    sampler.stop()
    # back-to-back launches without the flush (the features stay in L2, as
    # they would right after the verifier wrote them): about the kernel's own
    # duration per launch
    b2b, _, _ = timed_repeats(step, K, stream, dev, world, B, min_s=0.2)
    b2b_ms = statistics.median(b2b)
    # the same launches replayed from a CUDA graph (no host cost between them)
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gr, capture_error_mode="thread_local"):
        gs = torch.cuda.current_stream(dev)
        for _ in range(20):
            B.pr_quantile_score(ctx, feat, off, w, wl.tau, score=score, ship=ship,
                                req_flags=rflags, want_summary=False, stream=gs)
    for _ in range(3):
        gr.replay()
    torch.cuda.synchronize(dev)
    g_per, _, _ = timed_repeats(gr.replay, 10, torch.cuda.current_stream(dev), dev, world, B,
                                min_s=0.2)
    graph_ms = statistics.median(g_per) / 20
    del gr

    hf, ho = torch.from_numpy(feat_h).pin_memory(), torch.from_numpy(offsets).pin_memory()
    hs = torch.empty(n_req).pin_memory()
    hsh = torch.empty(n_req, dtype=torch.uint8).pin_memory()
    hfl = torch.empty(n_req, dtype=torch.int32).pin_memory()
    dfeat, doff = torch.empty_like(feat), torch.empty_like(off)

    def e2e_step():
        dfeat.copy_(hf, non_blocking=True)
        doff.copy_(ho, non_blocking=True)
        B.pr_quantile_score(ctx, dfeat, doff, w, wl.tau, score=score, ship=ship, req_flags=rflags,
                            want_summary=False, stream=stream)
        hs.copy_(score, non_blocking=True)
        hsh.copy_(ship, non_blocking=True)
        hfl.copy_(rflags, non_blocking=True)
        torch.cuda.synchronize(dev)

    e2e_step()
    e2e_steps = max(3, min(K, 50))
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    barrier(world)
    e2e_s = reduce_max(time.perf_counter() - t0, world, dev)

    qbytes = qnt_bytes(n_rows, n_req)
    peaks_file = os.path.join(ROOT, "MEASURED_PEAKS.json")
    peak = float(json.load(open(peaks_file))["hbm_gbs"]) if os.path.exists(peaks_file) else 6800.0
    achieved = qbytes / (ms / 1e3) / 1e9
    if rank == 0:
        out = subprocess.run([sys.executable, os.path.abspath(__file__), "--qnt-oracle-child",
                              "--q-layout", args.q_layout],
                             env=dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1",
                                      MKL_NUM_THREADS="1"),
                             capture_output=True, text=True, check=True)
        d = json.loads(out.stdout.strip().splitlines()[-1])
        so, po = np.asarray(d["score"]), np.asarray(d["ship"])
        g = score.cpu().numpy().astype(np.float64)
        ok = bool(np.all(np.abs(g - so) <= 1e-5) and
                  np.all((ship.cpu().numpy() == po) | (np.abs(so - wl.tau) < 1e-6)))
        print(json.dumps({
            "metric": "scored tokens/sec (quantile summary + MLP, %s)" % (
                "1,024-request ragged layout" if args.q_layout == "ragged" else
                "64-request full-response layout"),
            "value": n_rows * world / (ms / 1e3), "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": "quantile summary + MLP: %d requests, %s (%d rows), seeded "
                                   "feature records and weights (6,081 floats)" % (
                                       n_req, "lognormal lengths (median 128, 8..1,024)"
                                       if args.q_layout == "ragged" else "T~U{32..256}", n_rows),
                       "l2": "256 MB written between timed steps (flush)"},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak,
                         "unit": "GB/s", "frac": achieved / peak,
                         "traffic": profiled_file_traffic(QNT_PROFILE, QNT_FILES),
                         "kernel": "qmlp_requests",
                         "peak_source": "measured",
                         "note": "latency-bound: one CTA per request, 2.25 waves; the "
                                 "per-request chains (loads, rank or sort, MLP), not bandwidth, "
                                 "set the time",
                         "algorithmic_bytes_per_launch": qbytes, "avg_launch_ms": ms,
                         "back_to_back_launch_ms": b2b_ms,
                         "graph_launch_ms": graph_ms},
            "cpu_baseline": {"value": n_rows / d["seconds"], "unit": UNIT, "cores": 1,
                             "kind": "oracle",
                             "sample": "the whole %d-row workload, float64 numpy oracle" % n_rows},
            "e2e": {"value": n_rows * world * e2e_steps / e2e_s, "unit": UNIT,
                    "h2d_bytes_per_step": hf.numel() * 4 + ho.numel() * 8,
                    "d2h_bytes_per_step": n_req * 9,
                    "api": "pr_quantile_score with host copies of features, offsets and results"},
            "gpu_launches": launches,
            "clocks": clocks,
            "parity": {"requests_checked": n_req, "ok": ok},
        }))
    B.pr_ctx_destroy(ctx)
    return 0


SEL_FILES = ("pr_device.cuh", "pr_select.cuh", "pr_select_api.cu")
SEL_PROFILE = os.path.join(ROOT, "profiles", "sel_scatter_u32_pool16m.md")
SEL_N = 1 << 24


def sel_oracle_child(n: int):
    from oracle import selective as osel
    s, y = W.selective_pool(n)
    t0 = time.perf_counter()
    o = osel.selective_metrics(s, y, 0.5)
    dt = time.perf_counter() - t0
    print(json.dumps({"seconds": dt, "out": o}))
    return 0


def run_selective_workload(args):
    """Coverage calibration plus AUROC / AUARC on a 2^24-score validation pool
    (pr_selective_metrics): one radix sort and the metric scans per step."""
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2608_28726_gb300 import build as prbuild
    prbuild.build()
    from paper_2608_28726_gb300 import binding as B
    n, q = SEL_N, 0.5
    s_h, y_h = W.selective_pool(n)
    sc, lb = torch.from_numpy(s_h).to(dev), torch.from_numpy(y_h).to(dev)
    ctx = B.pr_ctx_create(local, max_rows=0, max_requests=1)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    K = args.steps
    res = {}

    def step():
        res["r"] = B.pr_selective_metrics(ctx, sc, q, labels=lb, stream=stream)

    sampler = ClockSampler(local)
    sampler.start()

    def timed(timing: int):
        B.pr_ctx_set_option(ctx, B.PR_OPT_TIMING, timing)
        for _ in range(max(3, args.warmup)):
            step()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(K)]
        kms = []
        barrier(world)
        torch.cuda.synchronize(dev)
        n0 = B.launch_count()
        for i in range(K):
            flush.zero_()
            ev[i][0].record(stream)
            step()
            ev[i][1].record(stream)
            if timing:
                kms.append(B.pr_ctx_kernel_times(ctx))
        torch.cuda.synchronize(dev)
        barrier(world)
        tot = sum(a.elapsed_time(b) for a, b in ev)
        return reduce_max(tot, world, dev) / K, B.launch_count() - n0, kms

    t_wall0 = time.time()
    ms, launches, _ = timed(0)
    t_wall1 = time.time()
    iso_ms, _, kms = timed(1)
    B.pr_ctx_set_option(ctx, B.PR_OPT_TIMING, 0)
    clocks = sampler.summary(t_wall0, t_wall1)
    sampler.stop()
    scatter_ms = float(np.mean([k[i] for k in kms for i in (3, 6, 9, 12)]))
    per_kernel = np.mean(np.asarray(kms), axis=0).tolist()
    got = res["r"]

    hs, hy = torch.from_numpy(s_h).pin_memory(), torch.from_numpy(y_h).pin_memory()
    ds, dy = torch.empty_like(sc), torch.empty_like(lb)

    def e2e_step():
        ds.copy_(hs, non_blocking=True)
        dy.copy_(hy, non_blocking=True)
        return B.pr_selective_metrics(ctx, ds, q, labels=dy, stream=stream)

    e2e_step()
    e2e_steps = max(3, min(K, 20))
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    barrier(world)
    e2e_s = reduce_max(time.perf_counter() - t0, world, dev)

    peaks_file = os.path.join(ROOT, "MEASURED_PEAKS.json")
    peak = float(json.load(open(peaks_file))["hbm_gbs"]) if os.path.exists(peaks_file) else 6800.0
    scatter_bytes = 10 * n  # read key + label, write key + label
    step_bytes = 80 * n
    achieved = scatter_bytes / (scatter_ms / 1e3) / 1e9
    if rank == 0:
        env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
        out = subprocess.run([sys.executable, os.path.abspath(__file__), "--sel-oracle-child",
                              str(n)], env=env, capture_output=True, text=True, check=True)
        d = json.loads(out.stdout.strip().splitlines()[-1])
        o = d["out"]
        ok = (got["k"] == o["k"] and got["n_ship"] == o["n_ship"] and
              got["n_finite"] == o["n_finite"] and got["n_pos"] == o["n_pos"] and
              np.float32(got["tau"]) == np.float32(o["tau"]) and
              abs(got["auroc"] - o["auroc"]) <= 1e-12 and abs(got["auarc"] - o["auarc"]) <= 1e-9)
        print(json.dumps({
            "metric": "validation scores calibrated and ranked per second (coverage tau, AUROC, "
                      "AUARC; 2^24-score pool)",
            "value": n * world / (ms / 1e3), "unit": "scores/s", "n_gpus": world, "steps": K,
            "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u32", "data": "synthetic",
            "config": {"workload": "selective metrics: %d seeded scores (sigmoid of N(0,1.5^2), "
                                   "1%% NaN), labels Bernoulli(score), q = %.2f" % (n, q),
                       "l2": "256 MB written between timed steps (flush)"},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak,
                         "traffic": profiled_file_traffic(SEL_PROFILE, SEL_FILES),
                         "kernel": "sel_scatter (radix pass)",
                         "algorithmic_bytes_per_launch": scatter_bytes,
                         "avg_launch_ms": scatter_ms,
                         "step_algorithmic_bytes": step_bytes,
                         "step_achieved_gbs": step_bytes / (ms / 1e3) / 1e9,
                         "isolated_kernel_ms": per_kernel, "isolated_step_ms": iso_ms},
            "cpu_baseline": {"value": n / d["seconds"], "unit": "scores/s", "cores": 1,
                             "kind": "oracle",
                             "sample": "the whole %d-score pool, float64 numpy oracle" % n},
            "e2e": {"value": n * world * e2e_steps / e2e_s, "unit": "scores/s",
                    "h2d_bytes_per_step": 5 * n, "d2h_bytes_per_step": 64,
                    "api": "pr_selective_metrics after host copies of scores and labels"},
            "gpu_launches": launches,
            "clocks": clocks,
            "parity": {"ok": bool(ok), "tau": got["tau"], "auroc": got["auroc"],
                       "auarc": got["auarc"]},
        }))
    B.pr_ctx_destroy(ctx)
    return 0


def run_prescore_workload(args):
    """The prompt pre-scorer of Eq. 2 on the host CPU (the paper keeps it off
    the accelerator): a vocabulary fitted on 20,000 seeded synthetic prompts,
    then batches of 100,000 prompts scored with all host threads."""
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from paper_2608_28726_gb300 import build as prbuild
    prbuild.build()
    from paper_2608_28726_gb300 import binding as B
    from oracle import prescore as op
    docs, _ = W.prompts(20000, seed=9401)
    prompts, images = W.prompts(100000, seed=9402)
    t0 = time.perf_counter()
    ps = B.pr_prescorer_fit(docs, min_df=2)
    fit_s = time.perf_counter() - t0
    V = B.pr_prescorer_vocab_size(ps)
    w, b = W.prescore_weights(V)
    cores = os.cpu_count() or 1
    import ctypes
    _buf, ptrs, _ = B._texts(prompts)  # the host arrays the C call reads, built once
    n = len(prompts)
    p_lib, z_lib = np.empty(n, np.float32), np.empty(n, np.float32)

    def call(n_threads=0, count=n):
        st = B._lib.pr_prescorer_score(ps, ptrs.ctypes.data, images.ctypes.data,
                                       count, w.ctypes.data, float(b), n_threads,
                                       p_lib.ctypes.data, z_lib.ctypes.data)
        assert st == 0, st

    for _ in range(max(1, args.warmup)):
        call()
    reps, t_start = [], time.perf_counter()
    while len(reps) < 3 or time.perf_counter() - t_start < MIN_TIMED_S:
        t0 = time.perf_counter()
        call()
        reps.append(time.perf_counter() - t0)
    sec = statistics.median(reps)
    t0 = time.perf_counter()
    call(n_threads=1, count=20000)
    one_core = 20000 / (time.perf_counter() - t0)
    # through the Python binding, its argument marshalling included
    t0 = time.perf_counter()
    p_api, _ = B.pr_prescorer_score(ps, prompts, images, w, b)
    api_sec = time.perf_counter() - t0
    call()
    # parity and the float64 oracle's own speed on a sample
    n_s = 2000
    m = op.fit(docs, min_df=2)
    t0 = time.perf_counter()
    p_or, z_or = op.score(m, prompts[:n_s], images[:n_s], w.astype(np.float64), b)
    oracle_s = time.perf_counter() - t0
    z_or = np.asarray(z_or)
    ok = bool(np.all(np.abs(z_lib[:n_s] - z_or) <= 1e-5 + 1e-6 * np.abs(z_or)) and
              np.all(np.abs(p_lib[:n_s] - np.asarray(p_or)) <= 1e-6) and
              np.array_equal(p_api, p_lib))
    text_bytes = sum(len(x) for x in prompts)
    B.pr_prescorer_destroy(ps)
    line = {
        "metric": "pre-scored prompts/sec (Eq. 2 prompt pre-scorer, host CPU)",
        "value": len(prompts) / sec, "unit": "prompts/s", "n_gpus": 0, "steps": len(reps),
        "warmup": max(1, args.warmup), "ms_per_step": sec * 1e3, "higher_is_better": True,
        "scaling": "none", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": "100,000 seeded synthetic prompts (mean %.0f bytes), vocabulary "
                               "of %d terms fitted on 20,000 others (min_df 2)" % (
                                   text_bytes / len(prompts), V),
                   "threads": cores, "fit_s": fit_s,
                   "note": "host CPU by design (Section 3.1 keeps the pre-scorer off the "
                           "accelerator): no GPU and no GPU roofline"},
        "roofline": {"bound": "host", "achieved": text_bytes / sec / 1e6, "unit": "MB/s of prompt "
                     "text", "peak": None, "frac": None, "one_core_prompts_per_s": one_core},
        "cpu_baseline": {"value": n_s / oracle_s, "unit": "prompts/s", "cores": 1,
                         "kind": "oracle", "sample": "prompts 0..%d, float64 Python oracle"
                                                     % (n_s - 1)},
        "e2e": {"value": len(prompts) / api_sec, "unit": "prompts/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0,
                "api": "binding.pr_prescorer_score from Python strings (encoding and "
                       "argument arrays included); value times the C call alone"},
        "gpu_launches": 0,
        "parity": {"prompts_checked": n_s, "ok": ok},
    }
    print(json.dumps(gate_on_parity(line)))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--workload", default=WORKLOAD,
                    choices=["full", "tiny", "ragged", "wide", "decode", "head", "selective",
                             "quantile", "lmhead", "prescore"],
                    help="full (default, the headline line), one of the other verifier "
                         "workloads, head (the transformer scorer head), quantile (the "
                         "quantile-summary MLP), selective (calibration and ranking metrics) "
                         "or lmhead (the LM head fused with the row reduction)")
    ap.add_argument("--configs", default="c1,c3,c4,c5",
                    help="default run: the other workloads measured into the line's `configs` "
                         "object (c1 tiny, c3 decode, c4 ragged, c5 wide; 'none' for none)")
    ap.add_argument("--requests", type=int, default=0,
                    help="profiling only: the first N requests of the workload")
    ap.add_argument("--timed-seconds", type=float, default=MIN_TIMED_S,
                    help="device time each timed measurement repeats its K-step loop for")
    ap.add_argument("--decode-steps", type=int, default=1000,
                    help="profiling only: the decode workload's first N steps (resident trace)")
    ap.add_argument("--skip-host", action="store_true",
                    help="profiling only: skip the host-memory and oracle legs")
    ap.add_argument("--head-oracle-sample", type=int, default=0, help=argparse.SUPPRESS)
    ap.add_argument("--head-layers", type=int, default=2, help=argparse.SUPPRESS)
    ap.add_argument("--sel-oracle-child", type=int, default=0, help=argparse.SUPPRESS)
    ap.add_argument("--qnt-oracle-child", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--q-layout", default="ragged", choices=sorted(Q_LAYOUTS),
                    help="quantile workload: the ragged (default) or full-response request layout")
    ap.add_argument("--lm-oracle-child", type=int, default=0, help=argparse.SUPPRESS)
    ap.add_argument("--lm-rows", type=int, default=0,
                    help="lmhead workload: the first N hidden states only, as one request")
    args = ap.parse_args()
    globals()["MIN_TIMED_S"] = args.timed_seconds
    if args.lm_oracle_child:
        return lm_oracle_child(args.lm_oracle_child)
    if args.qnt_oracle_child:
        return qnt_oracle_child(args.q_layout)
    if args.head_oracle_sample:
        return head_oracle_child(args.head_oracle_sample, args.head_layers)
    if args.sel_oracle_child:
        return sel_oracle_child(args.sel_oracle_child)
    if args.impl == "reference":
        return run_reference(args)
    if args.workload == "head":
        return run_head_workload(args)
    if args.workload == "selective":
        return run_selective_workload(args)
    if args.workload == "prescore":
        return run_prescore_workload(args)
    if args.workload == "quantile":
        return run_quantile_workload(args)
    if args.workload == "lmhead":
        return run_lmhead_workload(args)
    if args.workload != WORKLOAD:
        return run_other_workload(args)
    return run_gb300(args)


if __name__ == "__main__":
    sys.exit(main())
