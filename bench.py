"""Benchmark: masked decode steps on the 1024 x 262,144 C-like workload.

One step = one pass of the whole per-step path over the batch, psc_decode_step
(called as its two halves, psc_decode_step_mask + psc_decode_step_advance, so
that the masking kernel can be timed on its own; the same steps replayed from a
CUDA graph are reported beside the timed region):
  k_step_tma       apply every row's precomputed mask to the bf16 logits in
                   place, write the packed bitmask [B][V/32] and pick the greedy
                   token among the allowed ones, in one TMA-pipelined pass
                   (k_step_warp, a warp per 1024-column chunk, at small batches)
  k_advance_warp   lex + parse the chosen tokens on the device-resident stacks
                   and classify the new configurations (bottom-up classifier:
                   only the stack entries the step changed are re-read)

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
                       [--mode teacher | sweep]
For N > 1 launch with torch.distributed.run: every rank runs an independent
replica (the rows of different sequences are independent; no collective on the
data path) and the step rate is summed over ranks (weak scaling).
The reference arm (--impl reference) times the CPU oracle on the host cores.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = 5
SEQ = 32          # decode steps per sequence of the workload
METRIC = "masked decode steps/s and µs/step at batch×vocab; HBM GB/s vs GB300 peak"
UNIT = "steps/s"
PROFILE_FILE = os.path.join(ROOT, "profiles", "k_step_tma_c5_traffic.txt")


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ------------------------------------------------------------ clock sampling
class ClockSampler:
    """Samples SM clock and clock-event reasons through NVML (read-only) while
    the timed region runs; falls back to nvidia-smi."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, index: int = 0, period_s: float = 0.0005):
        self.samples = []
        self.reasons = set()
        self.max_mhz = None
        self.period = period_s
        self._stop = threading.Event()
        self._nvml = None
        self._proc = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() == 0:
                h = ctypes.c_void_p()
                if nv.nvmlDeviceGetHandleByIndex_v2(index, ctypes.byref(h)) == 0:
                    self._nvml, self._h = nv, h
                    mx = ctypes.c_uint()
                    if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
                        self.max_mhz = mx.value
        except OSError:
            self._nvml = None

    def _loop(self):
        nv, h = self._nvml, self._h
        clk, rs = ctypes.c_uint(), ctypes.c_ulonglong()
        get_r = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            nv.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self._stop.is_set():
            if nv.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0:
                self.samples.append(clk.value)
            if get_r(h, ctypes.byref(rs)) == 0:
                for bit, name in self.REASONS.items():
                    if rs.value & bit:
                        self.reasons.add(name)
            time.sleep(self.period)

    def __enter__(self):
        if self._nvml is not None:
            self._t = threading.Thread(target=self._loop, daemon=True)
            self._t.start()
        else:
            try:
                self._proc = subprocess.Popen(
                    ["nvidia-smi", "--query-gpu=clocks.sm,clocks.max.sm,clocks_event_reasons.active",
                     "--format=csv,noheader,nounits", "-lms", "50"],
                    stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            except OSError:
                self._proc = None
        return self

    def __exit__(self, *a):
        self._stop.set()
        if self._nvml is not None:
            self._t.join()
        elif self._proc is not None:
            self._proc.terminate()
            out = self._proc.communicate(timeout=5)[0]
            for line in out.splitlines():
                parts = [p.strip() for p in line.split(",")]
                try:
                    self.samples.append(int(parts[0]))
                    self.max_mhz = int(parts[1])
                    mask = int(parts[2], 16)
                    for bit, name in self.REASONS.items():
                        if mask & bit:
                            self.reasons.add(name)
                except (ValueError, IndexError):
                    pass

    def summary(self):
        return {"sm_mhz": statistics.median(self.samples) if self.samples else None,
                "sm_max_mhz": self.max_mhz, "reasons": sorted(self.reasons),
                "samples": len(self.samples)}


# ---------------------------------------------------------------- oracle arm
def oracle_rate(w, budget_s: float, threads: int):
    """Time the CPU oracle (as it stands) on whole rows of the workload until
    about budget_s seconds of wall time; returns (steps/s, rows, seconds)."""
    from oracle import Oracle, Vocab
    o = Oracle(w.grammar_text)
    voc = Vocab.from_list(w.vocab, w.eos_id)
    cfgs = []
    rows = 0
    spent = 0.0
    n = 1
    while spent < budget_s and rows < w.B:
        batch = []
        for b in range(rows, min(rows + n, w.B)):
            oc = o.initial()
            o.advance_tokens(oc, voc, w.prefix_ids[b])
            batch.append(oc)
        t0 = time.perf_counter()
        o.masks(batch, voc, threads=threads)
        spent += time.perf_counter() - t0
        rows += len(batch)
        cfgs.extend(batch)
        n *= 2
    return rows / (spent * w.B), rows, spent


def run_reference(args):
    """The reference arm: the CPU oracle as it stands, on the host cores.  A
    whole 1024-row step of the oracle takes tens of seconds, so each timed step
    is a bounded sample of the workload: the oracle's masks for one row (all V
    tokens), a different prefix row each step.  The line reports what was timed
    (rows_timed, us_per_row, ms_per_step = wall time per timed one-row step) and
    the metric in steps of the whole batch (value = rows per second / B)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from workloads import configs
    w = configs.load(WORKLOAD)
    threads = os.cpu_count() or 1
    from oracle import Oracle, Vocab
    o = Oracle(w.grammar_text)
    voc = Vocab.from_list(w.vocab, w.eos_id)
    cfgs = []
    for b in range(args.warmup + args.steps):
        oc = o.initial()
        o.advance_tokens(oc, voc, w.prefix_ids[b % w.B])
        cfgs.append(oc)
    for i in range(args.warmup):
        o.masks([cfgs[i]], voc, threads=threads)
    t0 = time.perf_counter()
    for i in range(args.steps):
        o.masks([cfgs[args.warmup + i]], voc, threads=threads)
    dt = time.perf_counter() - t0
    rows_per_s = args.steps / dt
    value = rows_per_s / w.B
    sample = (f"{args.steps} timed steps, each the oracle's masks for one of the {w.B} prefix rows "
              f"(rows {args.warmup}..{args.warmup + args.steps - 1}) x all {w.V} tokens on {threads} threads; "
              f"value = rows per second / {w.B}")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * dt / args.steps,
        "rows_timed": args.steps, "rows_per_step": 1, "us_per_row": dt / args.steps * 1e6,
        "ms_per_workload_step_extrapolated": 1000.0 / value,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32",
        "data": "synthetic", "config": config_block(w, args.gpus),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


# ------------------------------------------------------------- multi-rank
def max_over_ranks(x: float, device) -> float:
    """The largest x of all ranks (x itself with one process)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world: int, steps: int, elapsed_ms: float) -> float:
    """Steps/s of the whole job: every rank runs its own replica of the workload for
    the same number of steps; the slowest rank's time (max over ranks) counts."""
    return world * steps / (elapsed_ms / 1000.0)


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.barrier()


def config_block(w, n):
    return {"workload": f"config 5: C-like grammar, vocab {w.V}, batch {w.B}, bf16 logits ~N(0,2), "
                        "decode steps (mask+apply+greedy+advance)",
            "batch": w.B, "vocab": w.V, "logit_dtype": "bf16", "grammar": "synthetic C-like (150 rules)",
            "parallelism": f"replicas x{n}", "l2": "inputs larger than L2 (512 MiB logits per step)",
            "decode": f"sequences of {SEQ} greedy steps from the prefix states (restored from a device "
                      "copy before each sequence, inside the timed region); each step on its own logits "
                      "buffer"}


def code_only(src: str) -> str:
    """C/C++/CUDA source without its comments and blank lines (string and
    character literals kept as they are)."""
    out, i, n = [], 0, len(src)
    while i < n:
        c = src[i]
        if c in "\"'":
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        elif src.startswith("//", i):
            j = src.find("\n", i)
            i = n if j < 0 else j
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
            out.append(" ")
        else:
            out.append(c)
            i += 1
    return "\n".join(line.rstrip() for line in "".join(out).splitlines() if line.strip())


def device_source_hash() -> str:
    """sha256 of the device code of the library: psc_capi.cu up to its host glue
    and the headers it includes, comments left out, so host-only and comment-only
    edits keep the recorded traffic."""
    csrc = os.path.join(ROOT, "paper_2608_03065_gb300", "csrc")
    src = open(os.path.join(csrc, "psc_capi.cu"), encoding="utf-8").read()
    cut = src.find("// ----------------------------------------------------------------- host glue")
    h = hashlib.sha256(code_only(src[:cut] if cut > 0 else src).encode())
    for path in (os.path.join(csrc, "psc_internal.h"), os.path.join(ROOT, "include", "psc.h")):
        h.update(code_only(open(path, encoding="utf-8").read()).encode())
    return h.hexdigest()


def traffic_from_profile(kernel_src_hash: str):
    """Per-launch DRAM bytes of the fused kernel from the committed ncu summary,
    if it was taken on the current kernel source."""
    if not os.path.exists(PROFILE_FILE):
        return None
    vals = {}
    with open(PROFILE_FILE) as f:
        for line in f:
            if ":" in line:
                k, v = line.split(":", 1)
                vals[k.strip()] = v.strip()
    if vals.get("device_source_sha256") != kernel_src_hash:
        return None
    try:
        return int(vals["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


# ------------------------------------------------------------- teacher mode
def run_teacher(args):
    """RQ1: whole sentences of configs 2-4 are teacher-forced through the device
    path (psc_fill_mask, then psc_advance); the pass rate on them must be 1, and
    sentences with one random token spliced in are mostly stopped.  RQ2: one
    decoding step at batch 1 on the config-5 tables (mask + advance on the
    device), beside the same step through the library's host functions (the
    classifier walk, the mask-row copy and the parser step on the CPU)."""
    import numpy as np
    import torch
    from paper_2608_03065_gb300 import build, psc
    from workloads import configs, teacher
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    out = {"metric": "teacher-forced pass rate; batch-1 step latency", "mode": "teacher", "rq1": {}, "rq2": {}}

    def first_rejection(h, w, seqs):
        B = len(seqs)
        T = max(len(q) for q in seqs) + 1
        tokm = np.full((B, T), -1, dtype=np.int32)
        for b, q in enumerate(seqs):
            tokm[b, :len(q)] = q
            tokm[b, len(q)] = w.eos_id
        st = psc.psc_state_init(h, B, 256)
        bm = torch.empty(B, h.W, dtype=torch.int32, device=dev)
        first = np.full(B, -1, dtype=np.int64)
        for j in range(T):
            psc.psc_fill_mask(h, st, bm)
            m = bm.cpu().numpy().view(np.uint32)
            col = tokm[:, j]
            for b in np.nonzero((col >= 0) & (first < 0))[0]:
                v = int(col[b])
                if not ((m[b, v >> 5] >> (v & 31)) & 1):
                    first[b] = j
            psc.psc_advance(h, st, torch.from_numpy(np.where(first < 0, col, -1).astype(np.int32)).to(dev))
        torch.cuda.synchronize()
        return first, int(sum(len(q) + 1 for q in seqs))

    for cfg in (2, 3, 4):
        w = configs.load(cfg, batch=1)
        ts = teacher.teacher_set(w, 64)
        h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
        t0 = time.time()
        pos, ntok = first_rejection(h, w, ts.positives)
        neg, _ = first_rejection(h, w, ts.negatives)
        secs = time.time() - t0
        out["rq1"][w.spec.name] = {
            "sentences": len(ts.positives), "tokens": ntok,
            "positive_pass_rate": float((pos < 0).mean()),
            "negative_stopped_rate": float((neg >= 0).mean()),
            "stopped_before_splice": int(sum(1 for r, k in zip(neg, ts.inserted_at) if 0 <= r < k)),
            "wall_s": round(secs, 2)}

    # RQ2 on config 5's tables, one row
    w = configs.load(5, batch=1)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    ids = w.prefix_ids[0]
    n = min(len(ids), 200)
    st = psc.psc_state_init(h, 1, 256)
    bm = torch.empty(1, h.W, dtype=torch.int32, device=dev)
    toks = [torch.tensor([v], dtype=torch.int32, device=dev) for v in ids[:n]]
    stream = torch.cuda.current_stream()
    for i in range(5):
        psc.psc_fill_mask(h, st, bm, stream=stream)
    torch.cuda.synchronize()
    st = psc.psc_state_init(h, 1, 256)
    evs = []
    for i in range(n):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        psc.psc_fill_mask(h, st, bm, stream=stream)
        psc.psc_advance(h, st, toks[i], stream=stream)
        b.record(stream)
        evs.append((a, b))
    torch.cuda.synchronize()
    gpu_us = sorted(a.elapsed_time(b) * 1000.0 for a, b in evs)
    logits = [(torch.randn(1, w.V, device=dev) * w.spec.sigma).to(torch.bfloat16) for _ in range(8)]
    tok1 = torch.empty(1, dtype=torch.int32, device=dev)
    st2 = psc.psc_state_init(h, 1, 256)
    for v in ids[:20]:
        psc.psc_advance(h, st2, torch.tensor([v], dtype=torch.int32, device=dev))
    evs = []
    for i in range(64):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        psc.psc_decode_step(h, st2, logits[i % 8], tok1, stream=stream)
        b.record(stream)
        evs.append((a, b))
    torch.cuda.synchronize()
    dec_us = sorted(a.elapsed_time(b) * 1000.0 for a, b in evs)
    # host: the library's C functions called directly (ctypes call overhead included)
    lib = psc.load()
    hh = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True)
    cap = 256
    stack = np.zeros(cap, dtype=np.uint16)
    row = np.zeros(hh.W, dtype=np.uint32)
    q, depth, status = ctypes.c_int32(0), ctypes.c_int32(1), ctypes.c_int32(0)
    host_us = []
    for i in range(n):
        t0 = time.perf_counter()
        mid = lib.psc_host_classify(hh.ptr, q.value, stack.ctypes.data, depth.value, status.value)
        lib.psc_host_mask_row(hh.ptr, mid, row.ctypes.data)
        lib.psc_host_advance(hh.ptr, ctypes.byref(q), stack.ctypes.data, ctypes.byref(depth), cap,
                             ctypes.byref(status), int(ids[i]))
        host_us.append((time.perf_counter() - t0) * 1e6)
    host_us.sort()
    med = lambda a: round(a[len(a) // 2], 2)
    out["rq2"] = {"tables": w.spec.name, "steps": n,
                  "gpu_fill_mask_plus_advance_b1_us": {"median": med(gpu_us), "p90": round(gpu_us[int(0.9 * len(gpu_us))], 2)},
                  "gpu_decode_step_b1_us": {"median": med(dec_us), "vocab": w.V},
                  "host_walk_mask_row_advance_us": {"median": med(host_us), "note": "one CPU thread, ctypes call overhead included"}}
    print(json.dumps(out))


# --------------------------------------------------------------- sweep mode
def batch_points(psc, h, w, dev, batches, dtypes, n=16):
    """psc_decode_step on the workload's tables at the given batch sizes (rows
    0..B-1 of the prefix states) and logit types, two ways:
      graph: a CUDA graph holding the restore of the prefix states
        (psc_state_copy) and n decode steps on n logits buffers, replayed; µs per
        step = replay time / n (the device time of a step: no host calls between
        launches, as a decode loop captured in a graph runs);
      eager: each step called from Python between CUDA events (µs per step =
        median of n; at small batches this is the host's call latency).
    The rate of the formula's bytes is given for the graph time."""
    import torch
    V = w.V
    tm = torch.from_numpy(w.token_matrix()).to(dev)
    peak, _ = measured_peaks()
    stream = torch.cuda.current_stream()
    snaps = {}
    for B in batches:
        snaps[B] = psc.psc_state_init(h, B, 256)
        for j in range(tm.shape[1]):
            psc.psc_advance(h, snaps[B], tm[:B, j].contiguous())
    points = []
    for dt, esz in dtypes:
        for B in batches:
            st = psc.psc_state_init(h, B, 256)
            toks = [torch.empty(B, dtype=torch.int32, device=dev) for _ in range(n)]
            gen = torch.Generator(device=dev).manual_seed(B)
            xs = [(torch.randn(B, V, generator=gen, device=dev) * w.spec.sigma).to(dt) for _ in range(n)]
            for i in range(3):   # warm-up
                psc.psc_state_copy(st, snaps[B], stream=stream)
                psc.psc_decode_step(h, st, xs[i].clone(), toks[i], stream=stream)
            times = []
            for i in range(n):
                psc.psc_state_copy(st, snaps[B], stream=stream)
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                psc.psc_decode_step(h, st, xs[i], toks[i], stream=stream)
                b.record(stream)
                torch.cuda.synchronize()
                times.append(a.elapsed_time(b) * 1000.0)
            times.sort()
            eager = times[n // 2]
            # the same n steps captured once in a CUDA graph
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                cs = torch.cuda.current_stream()
                psc.psc_state_copy(st, snaps[B], stream=cs)
                for i in range(n):
                    psc.psc_decode_step(h, st, xs[i], toks[i], stream=cs)
            reps = []
            for r in range(8):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                g.replay()
                b.record(stream)
                torch.cuda.synchronize()
                if r >= 3:
                    reps.append(a.elapsed_time(b) * 1000.0 / n)
            graph = sorted(reps)[len(reps) // 2]
            alg = B * V // 8 + 2 * B * V * esz
            points.append({"dtype": "bf16" if esz == 2 else "f32", "batch": B,
                           "us_per_step_graph": round(graph, 2), "us_per_step_eager": round(eager, 2),
                           "algorithmic_GBps": round(alg / (graph * 1e-6) / 1e9, 1),
                           "frac": round(alg / (graph * 1e-6) / 1e9 / peak, 3)})
            del g, xs
            torch.cuda.empty_cache()
    return points


def run_sweep(args):
    """psc_decode_step on config 5's tables at batch 1, 16, 128 and 1024 with bf16
    and f32 logits (see batch_points)."""
    import torch
    from paper_2608_03065_gb300 import build, psc
    from workloads import configs
    build.build()
    dev = torch.device("cuda", 0)
    w = configs.load(WORKLOAD)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    pts = batch_points(psc, h, w, dev, (1, 16, 128, 1024), ((torch.bfloat16, 2), (torch.float32, 4)))
    print(json.dumps({"metric": "decode step over batch size and logit type", "mode": "sweep", "vocab": w.V,
                      "points": pts}))


# ------------------------------------------------------------- compile mode
def compile_one(cfg: int, vocab: int | None):
    """(child process) Compile one workload's tables on the host and print their
    sizes, the compile time and this process's peak RSS (nothing else runs in it)."""
    import resource
    import tempfile
    from paper_2608_03065_gb300 import build, psc
    from workloads import configs, sample
    build.build()
    spec = configs.SPECS[cfg]
    g = configs.grammar_spec(cfg)
    V = vocab or spec.V
    toks = configs.vocab_for(cfg, V)
    opts = dict(configs.COMPILE_LIMITS.get(cfg, {}))
    t0 = time.time()
    h = psc.psc_compile(g.text(), toks, len(toks) - 1, host_only=True, **opts)
    secs = time.time() - t0
    i = h.info()
    out = {"workload": spec.name if vocab is None else f"{spec.name.split('_v')[0]}_v{V}", "vocab": V,
           "compile_s": round(secs, 2), "threads": os.cpu_count(),
           "lalr_states": i.n_parser_states, "lexer_states": i.n_lexer_states,
           "states_built": i.states_built, "classifier_states": i.n_classifier_states,
           "classifier_layout": "sparse" if i.classifier_sparse else "dense",
           "classifier_bytes": i.classifier_bytes,
           "dense_classifier_bytes": i.n_classifier_states * i.n_parser_states * 4,
           "masks": i.n_masks, "mask_bytes": i.mask_bytes, "bottom_up_states": i.bottom_up_states,
           "bottom_up_bytes": i.bottom_up_bytes}
    with tempfile.TemporaryDirectory() as d:
        for codec in ("default", "none"):
            if codec == "none":
                os.environ["PSC_SAVE_CODEC"] = "none"
            path = os.path.join(d, f"{codec}.psc")
            t0 = time.time()
            psc.psc_save(h, path)
            with open(path, "rb") as f:
                head = f.read(12)
            key = "file_bytes" if codec == "default" else "file_bytes_uncompressed"
            out[key] = os.path.getsize(path)
            if codec == "default":
                out["codec"] = {0: "none", 1: "zstd", 2: "zlib"}[int.from_bytes(head[8:12], "little")]
                out["save_s"] = round(time.time() - t0, 2)
                t0 = time.time()
                psc.psc_load(path, host_only=True)
                out["load_s"] = round(time.time() - t0, 2)
    out["peak_rss_gb"] = round(resource.getrusage(resource.RUSAGE_SELF).ru_maxrss / 2**20, 2)
    print(json.dumps(out))


def graph_step_us(psc, h, w, B, n=16, cap=256):
    """Device time of one decode step at batch B on the workload's prefix states:
    a CUDA graph of n steps (psc_decode_step on n logits buffers), replayed."""
    import torch
    dev = torch.device("cuda", 0)
    tm = torch.from_numpy(w.token_matrix()).to(dev)
    snap = psc.psc_state_init(h, B, cap)
    for j in range(tm.shape[1]):
        psc.psc_advance(h, snap, tm[:B, j].contiguous())
    st = psc.psc_state_init(h, B, cap)
    gen = torch.Generator(device=dev).manual_seed(B)
    xs = [(torch.randn(B, w.V, generator=gen, device=dev) * w.spec.sigma).to(torch.bfloat16) for _ in range(n)]
    toks = [torch.empty(B, dtype=torch.int32, device=dev) for _ in range(n)]
    psc.psc_state_copy(st, snap)
    psc.psc_decode_step(h, st, xs[0].clone(), toks[0])
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        cs = torch.cuda.current_stream()
        psc.psc_state_copy(st, snap, stream=cs)
        for i in range(n):
            psc.psc_decode_step(h, st, xs[i], toks[i], stream=cs)
    reps = []
    for r in range(6):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        g.replay()
        b.record()
        torch.cuda.synchronize()
        if r >= 2:
            reps.append(a.elapsed_time(b) * 1000.0 / n)
    return round(sorted(reps)[len(reps) // 2], 2)


def run_compile(args):
    """Construction at scale (the paper's preprocessing cost and runtime memory,
    Section 5, Tables 6 and 7, report the same quantities for its Python
    implementation): each workload compiled in its own process on the host cores
    (compile time, peak RSS, classifier and mask sizes, saved file sizes); then,
    on the GPU, the decode step on the Java-sized tables at 4,096 and 262,144
    tokens (sparse classifier, packed parser tables staged in shared memory; also
    with the parser tables read from global memory, and at 262,144 tokens with
    stacks walked from the top instead of the bottom-up classifier) and on the
    262,144-token C-like
    tables with the advance's tables staged in shared memory or read from
    global memory."""
    jobs = [(2, None), (3, None), (4, None), (5, None), (6, 1024), (6, 2048), (6, 4096), (7, 131072), (7, None),
            (8, 32768), (8, None)]
    if args.steps > 1000:   # --steps above 1000: also the 8,192-token Java-sized vocabulary
        jobs.append((6, 8192))
    rows = []
    for cfg, voc in jobs:
        cmd = [sys.executable, os.path.abspath(__file__), "--mode", "compile-one", "--cfg", str(cfg)]
        if voc:
            cmd += ["--vocab", str(voc)]
        r = subprocess.run(cmd, capture_output=True, text=True)
        line = [x for x in r.stdout.splitlines() if x.startswith("{")]
        rows.append(json.loads(line[-1]) if r.returncode == 0 and line else
                    {"workload": f"config {cfg} vocab {voc}", "error": (r.stderr or r.stdout)[-400:]})
    out = {"mode": "compile", "metric": "construction time, peak RSS and table sizes", "compile": rows}
    try:
        import torch
        if torch.cuda.is_available():
            from paper_2608_03065_gb300 import build, psc
            from workloads import configs
            build.build()
            import tempfile
            for cfg, key, opts in ((6, "java_like_decode_step_us", {"bottom_up": False}),
                                   (7, "java_like_pretok_262144_decode_step_us", {}),
                                   (8, "sql_like_pretok_128256_decode_step_us", {"bottom_up": False})):
                w = configs.load(cfg)
                h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, **opts, **configs.COMPILE_LIMITS[cfg])
                i = h.info()
                rec = {"batch": w.B, "vocab": w.V, "classifier_sparse": i.classifier_sparse,
                       "bottom_up_states": i.bottom_up_states, "advance_table_bytes": i.advance_table_bytes,
                       "advance_tables_packed": i.advance_tables_packed,
                       "graph_us": graph_step_us(psc, h, w, w.B)}
                with tempfile.TemporaryDirectory() as d:
                    path = os.path.join(d, "t.psc")
                    psc.psc_save(h, path)
                    del h
                    hg = psc.psc_load(path, global_tables=True, bottom_up=opts.get("bottom_up", True))
                    rec["graph_us_global_tables"] = graph_step_us(psc, hg, w, w.B)
                    del hg
                    if cfg == 7:
                        ht = psc.psc_load(path, bottom_up=False)
                        rec["graph_us_top_down"] = graph_step_us(psc, ht, w, w.B)
                        del ht
                out[key] = rec
            w5 = configs.load(5)
            for gt in (False, True):
                h5 = psc.psc_compile(w5.grammar_text, w5.vocab, w5.eos_id, global_tables=gt)
                out.setdefault("c_like_262144_decode_step_us", {})[
                    "global_tables" if gt else "staged_tables"] = graph_step_us(psc, h5, w5, w5.B)
                del h5
    except Exception as e:   # the construction numbers stand without a GPU
        out["gpu_error"] = str(e)[:300]
    print(json.dumps(out))


# ------------------------------------------------------------- profile mode
def run_profile(args):
    """A small case for profiler captures: the workload's tables and prefix states,
    then three decode steps (psc_decode_step_mask + psc_decode_step_advance) on
    fresh logits, each inside an NVTX range named "decode" (config 5 by default, about
    2 GB on the device; --cfg picks another workload)."""
    import torch
    from paper_2608_03065_gb300 import build, psc
    from workloads import configs
    build.build()
    w = configs.load(args.cfg)
    opts = dict(configs.COMPILE_LIMITS.get(args.cfg, {}))
    if args.cfg in (6, 8):
        opts["bottom_up"] = False   # over its construction budget on these grammars and vocabularies
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, **opts)
    st = psc.psc_state_init(h, w.B, 256)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(h, st, tm[:, j].contiguous())
    g = torch.Generator(device="cuda").manual_seed(3)
    xs = [(torch.randn(w.B, w.V, generator=g, device="cuda") * w.spec.sigma).to(torch.bfloat16) for _ in range(3)]
    bm = torch.empty(w.B, h.W, dtype=torch.int32, device="cuda")
    tok = torch.empty(w.B, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    for i in range(3):
        torch.cuda.nvtx.range_push("decode")
        psc.psc_decode_step_mask(h, st, xs[i], bm)
        psc.psc_decode_step_advance(h, st, tok)
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_pop()
    print(json.dumps({"mode": "profile", "steps": 3, "rows_with_a_token": int((tok >= 0).sum())}))


def run_paths(args):
    """A small case for profiler captures of the plain mask paths on config 5's
    tables and prefix states (one 512 MiB logits buffer), each in an NVTX range:
    "fill_apply" (psc_fill_apply: masks applied from the current mask ids,
    k_apply_rows), "fill_mask" (psc_fill_mask, k_fill), "apply_mask"
    (psc_apply_mask from that bitmask, k_apply_rows), "classify_walk"
    (psc_fill_apply_noalloc on the same rows as plain arrays: every stack walked
    from the top by k_classify, then k_apply_rows), "classify_bottom_up" (a
    psc_advance with no tokens: every row classified again through its kept
    bottom-up states)."""
    import numpy as np
    import torch
    from paper_2608_03065_gb300 import build, psc
    from workloads import configs
    build.build()
    w = configs.load(WORKLOAD)
    B, V = w.B, w.V
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    st = psc.psc_state_init(h, B, 256)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(h, st, tm[:, j].contiguous())
    rows = psc.psc_states_download(st)
    q = torch.from_numpy(rows["q"]).cuda()
    depth = torch.from_numpy(rows["depth"]).cuda()
    status = torch.from_numpy(rows["status"]).cuda()
    stack = torch.from_numpy(rows["stack"].view(np.int16)).cuda()
    g = torch.Generator(device="cuda").manual_seed(9)
    x = (torch.randn(B, V, generator=g, device="cuda") * w.spec.sigma).to(torch.bfloat16)
    bm = torch.empty(B, h.W, dtype=torch.int32, device="cuda")
    none = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    steps = [("fill_apply", lambda: psc.psc_fill_apply(h, st, x, bm)),
             ("fill_mask", lambda: psc.psc_fill_mask(h, st, bm)),
             ("apply_mask", lambda: psc.psc_apply_mask(x, bm, B, V)),
             ("classify_walk", lambda: psc.psc_fill_apply_noalloc(h, q, depth, status, stack, x)),
             ("classify_bottom_up", lambda: psc.psc_advance(h, st, none))]
    for name, fn in steps:
        torch.cuda.nvtx.range_push(name)
        fn()
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_pop()
    print(json.dumps({"mode": "paths", "ranges": [n for n, _ in steps]}))


# ------------------------------------------------------------------ main arm
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=128)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cfg", type=int, default=WORKLOAD)
    ap.add_argument("--vocab", type=int, default=0)
    ap.add_argument("--mode", default="decode", choices=["decode", "teacher", "sweep", "profile", "paths", "compile",
                                                         "compile-one"],
                    help="decode: the benchmark line; teacher: teacher-forcing pass rates and "
                         "batch-1 step latency (the paper's RQ1/RQ2 measurements on these workloads); "
                         "sweep: decode-step time over batch sizes and logit types on config 5's tables; "
                         "profile: three decode steps in NVTX ranges, a small case for profiler captures; "
                         "paths: the plain mask paths (fill_apply, fill_mask, apply_mask, classification) in "
                         "NVTX ranges, for profiler captures; "
                         "compile: construction time, peak RSS and table sizes at real-grammar scale")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.mode == "teacher":
        return run_teacher(args)
    if args.mode == "sweep":
        return run_sweep(args)
    if args.mode == "profile":
        return run_profile(args)
    if args.mode == "paths":
        return run_paths(args)
    if args.mode == "compile":
        return run_compile(args)
    if args.mode == "compile-one":
        return compile_one(args.cfg, args.vocab or None)

    import torch
    import torch.distributed as dist
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)

    from paper_2608_03065_gb300 import build, psc
    from workloads import configs
    build.build()
    w = configs.load(WORKLOAD)
    B, V = w.B, w.V
    t0 = time.time()
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    compile_s = time.time() - t0
    info = h.info()
    st = psc.psc_state_init(h, B, 256)
    tm = torch.from_numpy(w.token_matrix()).to(dev)
    for j in range(tm.shape[1]):
        psc.psc_advance(h, st, tm[:, j].contiguous())
    torch.cuda.synchronize()

    # the workload's decode sequences: SEQ steps from the prefix states, which are
    # restored from a device copy before every sequence (the copy is timed too)
    snap = psc.psc_state_init(h, B, 256)
    psc.psc_state_copy(snap, st)
    K, Wm = args.steps, args.warmup
    n_buf = K + Wm
    gen = torch.Generator(device=dev).manual_seed(1000 * WORKLOAD + 4 + rank)
    sigma = w.spec.sigma
    bufs = [(torch.randn(B, V, generator=gen, device=dev) * sigma).to(torch.bfloat16) for _ in range(n_buf)]
    bitmask = torch.empty(B, h.W, dtype=torch.int32, device=dev)
    tok = torch.empty(B, dtype=torch.int32, device=dev)
    stat = torch.empty(B, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()
    # per-launch events on the first sequence only: an event between two kernels stops the
    # second from starting while the first finishes (programmatic dependent launch)
    n_ev = min(K, SEQ)
    ev = [tuple(torch.cuda.Event(enable_timing=True) for _ in range(3)) for _ in range(n_ev)]

    def step(i, timed=None, cs=None):
        cs = stream if cs is None else cs
        x = bufs[i]
        if timed is not None:
            ev[timed][0].record(cs)
        psc.psc_decode_step_mask(h, st, x, bitmask, stream=cs)
        if timed is not None:
            ev[timed][1].record(cs)
        psc.psc_decode_step_advance(h, st, tok, stat, stream=cs)
        if timed is not None:
            ev[timed][2].record(cs)

    def restore(cs=None):
        psc.psc_state_copy(st, snap, stream=stream if cs is None else cs)

    restore()
    for i in range(Wm):
        step(i)
    # per-kernel times: one decode sequence with CUDA events between the kernels (an event
    # between two kernels stops the second from starting during the first one's tail)
    restore()
    for i in range(n_ev):
        step(Wm + i, timed=i)
    torch.cuda.synchronize()
    # the same K steps (restores included, each step on its own logits buffer) captured once
    # in a CUDA graph and replayed (reported beside the timed region: at this batch the GPU
    # is the bottleneck either way)
    graph = torch.cuda.CUDAGraph()
    torch.cuda.synchronize()
    with torch.cuda.graph(graph):
        cs = torch.cuda.current_stream()
        for i in range(K):
            if i % SEQ == 0:
                restore(cs)
            step(Wm + i, cs=cs)
    torch.cuda.synchronize()
    g_a, g_b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g_a.record(stream)
    graph.replay()
    g_b.record(stream)
    torch.cuda.synchronize()
    graph_ms = max_over_ranks(g_a.elapsed_time(g_b), dev)
    del graph
    # the timed region: the K steps called one at a time
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(index=local) as clocks:
        torch.cuda.nvtx.range_push("psc_steps")
        t_start.record(stream)
        for i in range(K):
            if i % SEQ == 0:
                restore()
            step(Wm + i)
        t_end.record(stream)
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_pop()
    barrier()
    torch.cuda.synchronize()
    elapsed_ms = t_start.elapsed_time(t_end)
    mask_ms = [a.elapsed_time(b) for a, b, _ in ev]      # the masking kernel alone
    step_ms = [a.elapsed_time(c) for a, _, c in ev]      # the whole decode step
    elapsed_ms = max_over_ranks(elapsed_ms, dev)
    ms_per_step = elapsed_ms / K
    value = whole_job_rate(world, K, elapsed_ms)

    # end to end through the public API with host buffers: H2D of each step's
    # logits from pinned memory, the step, D2H of the chosen tokens.  Two device
    # buffers: the next step's logits are copied (on a second stream) while the
    # current step runs, as a serving loop would overlap them.
    n_host = 2
    host = [torch.empty(B, V, dtype=torch.bfloat16, pin_memory=True) for _ in range(n_host)]
    for k in range(n_host):
        host[k].copy_(bufs[k])
    tok_host = torch.empty(B, dtype=torch.int32, pin_memory=True)
    dbufs = [bufs[0], bufs[1]]
    copy_stream = torch.cuda.Stream(device=dev)
    ready = [torch.cuda.Event() for _ in range(2)]
    free = [torch.cuda.Event() for _ in range(2)]
    torch.cuda.synchronize()
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for k in range(2):
        free[k].record(stream)
    copy_stream.wait_stream(stream)
    with torch.cuda.stream(copy_stream):
        dbufs[0].copy_(host[0], non_blocking=True)
    ready[0].record(copy_stream)
    for i in range(K):
        cur, nxt = i % 2, (i + 1) % 2
        if i + 1 < K:   # the next step's logits, into the buffer the previous step used
            copy_stream.wait_event(free[nxt])
            with torch.cuda.stream(copy_stream):
                dbufs[nxt].copy_(host[(i + 1) % n_host], non_blocking=True)
            ready[nxt].record(copy_stream)
        if i % SEQ == 0:
            restore()
        stream.wait_event(ready[cur])
        psc.psc_decode_step(h, st, dbufs[cur], tok, bitmask, stat, stream=stream)
        free[cur].record(stream)
        tok_host.copy_(tok, non_blocking=True)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), dev)
    e2e_value = whole_job_rate(world, K, e2e_ms)

    # the plain mask paths on the same workload (prefix states, mask ids current),
    # each the median of 50 launches with CUDA events, logits buffers in rotation
    def median_us(fn, n=50):
        times = []
        for i in range(n):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn(bufs[i % n_buf])
            b.record(stream)
            times.append((a, b))
        torch.cuda.synchronize()
        return statistics.median(a.elapsed_time(b) * 1000.0 for a, b in times)

    restore()
    no_tokens = torch.full((B,), -1, dtype=torch.int32, device=dev)
    paths = {
        "fill_apply_us": median_us(lambda x: psc.psc_fill_apply(h, st, x, bitmask, stream=stream)),
        "fill_mask_us": median_us(lambda x: psc.psc_fill_mask(h, st, bitmask, stream=stream)),
        "apply_mask_us": median_us(lambda x: psc.psc_apply_mask(x, bitmask, B, V, stream=stream)),
        # a no-op advance still classifies every row: the classifier walk alone (+ launch)
        "classify_us": median_us(lambda x: psc.psc_advance(h, st, no_tokens, stream=stream)),
    }

    # small batches (decode latency): psc_decode_step at batch 1, 16 and 128 on the same tables
    small = batch_points(psc, h, w, dev, (1, 16, 128), ((torch.bfloat16, 2),))

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    peak, peak_kind = measured_peaks()
    alg_bytes = B * V // 8 + 2 * B * V * 2
    mask_avg_ms = sum(mask_ms) / len(mask_ms)
    step_avg_ms = sum(step_ms) / len(step_ms)
    achieved = alg_bytes / (mask_avg_ms / 1000.0) / 1e9
    traffic = traffic_from_profile(device_source_hash())

    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        threads = os.cpu_count() or 1
        rate, rows, secs = oracle_rate(w, 10.0, threads)
        rate1, rows1, secs1 = oracle_rate(w, 3.0, 1)
        cpu = {"value": rate, "unit": UNIT, "cores": threads, "kind": "oracle",
               "sample": f"oracle masks of the first {rows} of {w.B} rows x all {V} tokens "
                         f"({secs:.1f} s wall on {threads} threads), scaled to one {w.B}-row step",
               "us_per_row": secs / rows * 1e6,
               "single_thread": {"value": rate1, "unit": UNIT, "cores": 1, "us_per_row": secs1 / rows1 * 1e6,
                                 "sample": f"the first {rows1} rows ({secs1:.1f} s wall on 1 thread)"}}

    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": Wm,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "u32", "data": "synthetic", "config": config_block(w, world),
        "us_per_step": ms_per_step * 1000.0,
        "timing": "the K steps called one at a time between CUDA events; per-kernel times from a separate "
                  "decode sequence with events between the kernels",
        "graph": {"value": whole_job_rate(world, K, graph_ms), "unit": UNIT, "ms_per_step": graph_ms / K,
                  "note": "the same K steps captured once in a CUDA graph and replayed"},
        "decode_step_us": step_avg_ms * 1000.0,
        "k_step_tma_us": mask_avg_ms * 1000.0,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     # the same duration over the DRAM bytes ncu measured for one launch (the
                     # kernel skips bytes the formula counts: frac can pass 1, this cannot)
                     "dram_achieved": traffic / (mask_avg_ms / 1000.0) / 1e9 if traffic else None,
                     "dram_frac": traffic / (mask_avg_ms / 1000.0) / 1e9 / peak if traffic else None,
                     "kernel": "k_step_tma (masking pass + greedy choice, CUDA events around each launch)",
                     "algorithmic_bytes": alg_bytes, "peak_kind": peak_kind},
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": B * V * 2,
                "d2h_bytes_per_step": B * 4},
        "gpu_launches": 2 * K + (K + SEQ - 1) // SEQ,   # two per step, one per restore (k_state_copy)
        "clocks": clocks.summary(),
        "cpu_baseline": cpu,
        "mask_paths": paths,
        "small_batch": {"points": small, "note": "psc_decode_step (masking pass + greedy choice + advance) at "
                        "batch 1/16/128 on the same tables, bf16: graph = a CUDA graph of a prefix-state restore "
                        "and 16 steps on 16 logits buffers, replayed, time / 16 (the device time of a step); "
                        "eager = median of 16 steps called one at a time between CUDA events (host call latency "
                        "included)"},
        "device_timeouts": h.info().device_timeouts,
        "tables": {"classifier_states": info.n_classifier_states, "masks": info.n_masks,
                   "classifier_bytes": info.classifier_bytes, "mask_bytes": info.mask_bytes,
                   "compile_seconds": compile_s},
    }
    print(json.dumps(out))
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
