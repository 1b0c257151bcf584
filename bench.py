#!/usr/bin/env python
"""Benchmark of the SemPIC cache-hit path on GB300.

A step is one cache-hit pass over the workload up to the first token --
compose (layout + slot map), relocate (re-rotate + stitch, every layer), and
for every layer the inline append and the prefill attention -- the timer
boundary the paper defines for cache-hit TTFT, minus the Reader's linear and
MLP layers (no weights here).  Decode steps lie outside that boundary; when
the workload has decode tokens, one decode step over every layer is timed in
the same run and reported under rows.a6_decode.

Metric: cache-hit prefill query tokens per second (whole job), with the
per-kernel rooflines (relocate GB/s vs HBM, prefill attention TF/s vs bf16
tensor peak) in the same JSON line.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
       python bench.py --impl reference ...   (the CPU oracle, timed on the host)
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
GPU_GEN = {"tiny": "cpu", "llama8b_1layer": "cpu"}   # small inputs: CPU generator


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="stress_128k_b4",
                    help="default: the largest single-GPU workload (4 requests of ~139k tokens)")
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--prefill-splits", type=int, default=0)
    ap.add_argument("--decode-splits", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--layer-rope", action="store_true",
                    help="a rotary table per layer (bases 1e4 and the workload's, alternating)")
    ap.add_argument("--deviation", action="store_true",
                    help="also time the attention-deviation diagnostic on layer 0")
    ap.add_argument("--fused", action="store_true",
                    help="also time the rotate-on-load pass (default for stress_128k_b4)")
    ap.add_argument("--floor", action="store_true",
                    help="also time empty kernels with the pass's launch shapes (launch floor)")
    ap.add_argument("--oracle-sample", default=None, help=argparse.SUPPRESS)
    ap.add_argument("--oracle-seconds", type=float, default=10.0, help=argparse.SUPPRESS)
    ap.add_argument("--oracle-passes", type=int, default=0, help=argparse.SUPPRESS)
    return ap.parse_args(argv)


# ---------------------------------------------------------------- helpers
def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def src_sha(name):
    with open(os.path.join(ROOT, "paper_2607_28069_gb300", "csrc", name), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def max_over_ranks(x: float, world: int, device) -> float:
    """The largest value of x over the ranks of the job (x itself when alone):
    the job's time is its slowest rank's."""
    if world <= 1:
        return x
    import torch
    t = torch.tensor([x], device=device, dtype=torch.float64)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_step: float, steps: int, world: int, total_ms: float) -> float:
    """Whole-job throughput: the units every rank processed (each rank runs its
    own replica of the step) over the slowest rank's time."""
    return units_per_step * steps * world / (total_ms / 1e3)


def ncu_traffic(kernel_key, src_file):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current source of the kernel; else None."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(kernel_key)
    if not e or e.get("src_sha") != src_sha(src_file):
        return None
    return e.get("bytes_per_launch")


class ClockSampler:
    """SM clock and clock-event reasons sampled every ~1 ms during the timed
    region through NVML (the driver's library, via ctypes); nvidia-smi every
    200 ms when NVML is unavailable."""
    REASONS = {0x8: "hw_slowdown", 0x40: "hw_thermal_slowdown", 0x20: "sw_thermal_slowdown",
               0x4: "sw_power_cap", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, torch_device):
        self.dev = torch_device
        self.samples = []
        self.max_mhz = None
        self.source = None
        self._stop = None

    def _nvml_open(self):
        import ctypes
        import torch
        nvml = ctypes.CDLL("libnvidia-ml.so.1")
        if nvml.nvmlInit_v2() != 0:
            raise OSError("nvmlInit failed")
        h = ctypes.c_void_p()
        uuid = "GPU-" + str(torch.cuda.get_device_properties(self.dev).uuid)
        if nvml.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(h)) != 0:
            raise OSError("no NVML handle for " + uuid)
        mx = ctypes.c_uint()
        if nvml.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
            self.max_mhz = float(mx.value)
        fn = getattr(nvml, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            getattr(nvml, "nvmlDeviceGetCurrentClocksThrottleReasons")
        return nvml, h, fn

    def __enter__(self):
        import threading
        self._stop = threading.Event()
        try:
            nvml, h, reasons_fn = self._nvml_open()
            self.source = "nvml"

            def loop():
                import ctypes
                clk, rs = ctypes.c_uint(), ctypes.c_ulonglong()
                while not self._stop.is_set():
                    if nvml.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0 and \
                            reasons_fn(h, ctypes.byref(rs)) == 0:
                        self.samples.append((float(clk.value), int(rs.value)))
                    time.sleep(0.001)
            self._t = threading.Thread(target=loop, daemon=True)
            self._t.start()
        except (OSError, AttributeError):
            self.source = "nvidia-smi"
            self._proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=clocks.sm,clocks.max.sm,clocks_event_reasons.active",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        return self

    def __exit__(self, *exc):
        self._stop.set()
        if self.source == "nvml":
            self._t.join(timeout=2)
        elif self.source == "nvidia-smi":
            self._proc.terminate()
            out, _ = self._proc.communicate(timeout=5)
            for line in out.splitlines():
                parts = [x.strip() for x in line.split(",")]
                try:
                    self.samples.append((float(parts[0]), int(parts[2], 16)))
                    self.max_mhz = float(parts[1])
                except (ValueError, IndexError):
                    pass

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": ["unsampled"],
                    "source": self.source}
        seen = 0
        for _, r in self.samples:
            seen |= r
        return {"sm_mhz": statistics.median(c for c, _ in self.samples),
                "sm_max_mhz": self.max_mhz,
                "reasons": sorted(v for k, v in self.REASONS.items() if seen & k),
                "samples": len(self.samples), "source": self.source}


# ---------------------------------------------------------- work accounting
def work_of(spec, st):
    """Algorithmic work of one TTFT pass (and one decode step), from the
    request description (``workloads.Structure``): bytes for the HBM-bound
    rows, FLOPs for attention.  An inline token (prefix, post-document span
    or query) at logical position p sees the p + 1 keys before and at it."""
    L, Hq, Hkv, d = spec.layers, spec.q_heads, spec.kv_heads, spec.head_dim
    lens = [int(x) for x in st.lens]
    doc_tokens = sum(sum(lens[i] for i in docs) for docs in st.docs)
    pairs = 0
    query_tokens = 0
    inline_tokens = 0
    ctx = []
    for b, docs in enumerate(st.docs):
        P = st.prefixes[b]
        spans = st.spans[b]
        Tq = spec.query_len
        pairs += P * (P + 1) // 2                       # prefix rows see the prefix
        pos = P
        for i, s in zip(docs, spans):
            pos += lens[i]                              # the document, then its span
            pairs += s * pos + s * (s + 1) // 2
            pos += s
        pairs += Tq * pos + Tq * (Tq + 1) // 2          # query rows see all before them
        ctx.append(pos + Tq)
        query_tokens += Tq
        inline_tokens += P + sum(spans) + Tq
    row_bytes = Hkv * d * 2
    return {
        "query_tokens": query_tokens,
        "relocate_bytes": 4 * row_bytes * doc_tokens * L,               # K,V read + write
        "append_bytes": inline_tokens * (2 * Hq * d * 2 + 4 * row_bytes) * L,
        "attend_flops": 4 * d * Hq * pairs * L,                         # QK^T and PV
        "decode_bytes": sum(2 * row_bytes * (c + 1) for c in ctx) * L,  # K,V of step 0
        "ctx": ctx,
    }


METRIC = ("cache-hit prefill query tok/s (TTFT path: compose + relocate + append + prefill "
          "attention, all layers)")


def bench_config(workload, world):
    """The ``config`` object of the JSON line, the same for both arms: the
    workload by name and shape, computed from its selections alone."""
    from paper_2607_28069_gb300.workloads import WORKLOADS, draw_structure
    spec = WORKLOADS[workload]
    work = work_of(spec, draw_structure(spec))
    return {"workload": workload, "description": spec.description,
            "batch": spec.batch, "layers": spec.layers, "q_heads": spec.q_heads,
            "kv_heads": spec.kv_heads, "head_dim": spec.head_dim,
            "query_len": spec.query_len, "ctx_tokens": work["ctx"],
            "l2_policy": "L2 flushed before every step (a write of max(2 x L2, 256 MiB))",
            "timing": "value: one CUDA graph per pass, CUDA events at its two ends only; rows: "
                      "a second graph with event nodes at every call boundary, run in "
                      "alternate steps",
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU"}


# ------------------------------------------------------------- oracle arms
ORACLE_ROWS = 32   # query rows timed per oracle pass when a request has more
ORACLE_DOCS = 8    # documents re-rotated per oracle pass when a request has more


def oracle_sample(workload, seconds, passes=0):
    """Time the CPU oracle on bounded samples of the workload.

    A full oracle pass is one request through one layer: the layout
    (compose_layout), the re-rotation of every document (relocate_docs), the
    inline tokens' RoPE (rotary), the prefix rows' attention over the prefix
    and the query rows' attention over the whole stitched context
    (attention).  A sample times the layout, the inline RoPE and the prefix
    rows in full, and of the two large parts a seeded subset: ORACLE_DOCS of
    the request's documents (their time scaled by the request's document
    tokens over theirs) and ORACLE_ROWS of its query rows over the full
    context (scaled by query_len / ORACLE_ROWS; every query row sees the
    whole context, so their costs are equal).  The stitched context the
    attention reads is built once per request, untimed; requests of 50k
    positions or more use request 0 only (their set-up alone takes minutes).  Samples run until `seconds`
    elapse, or exactly `passes` of them.  Returns the per-sample estimates
    of a full pass and the rate in query tokens per second of the full
    workload (a request needs every layer)."""
    import dataclasses

    import numpy as np

    import oracle as O
    from paper_2607_28069_gb300.workloads import WORKLOADS, generate
    full = WORKLOADS[workload]
    # same selections and shapes per layer; one layer is enough for a sample
    spec = dataclasses.replace(full, layers=1, decode_steps=0)
    wl = generate(spec, device="cpu", gen_device="cpu")
    theta = O.rope_frequencies(spec.head_dim, spec.rope_base)
    f64 = lambda t: t.float().numpy().astype("float64")  # noqa: E731
    starts, lens = wl.doc_token_start.numpy(), wl.doc_len.numpy()
    base = wl.doc_base_pos.numpy()
    rng = np.random.default_rng(28069)
    Tq = spec.query_len
    ctx = {}

    def request(b):
        """Untimed set-up of request b: its inputs and its stitched context."""
        if b not in ctx:
            docs = wl.meta["docs"][b]
            tin = int(wl.inline_len[b])
            k_docs = [f64(wl.k_pool[0, starts[x]:starts[x] + lens[x]]) for x in docs]
            v_docs = [f64(wl.v_pool[0, starts[x]:starts[x] + lens[x]]) for x in docs]
            q, k, v = (f64(t[0, b, :tin]) for t in (wl.q_inline, wl.k_inline, wl.v_inline))
            lay = O.compose_layout(lens, base, docs, int(wl.prefix_len[b]), Tq,
                                   wl.block_table[b].numpy(), spec.page_size,
                                   span_len=wl.meta["spans"][b])
            K, V = O.dense_context(lay, k_docs, v_docs, base, k, v, theta)
            ctx[b] = (docs, k_docs, v_docs, q, k, K, V)
        return ctx[b]

    per_pass, b = [], 0
    while (passes and len(per_pass) < passes) or (not passes and (sum(per_pass) < seconds
                                                                  or not per_pass)):
        docs, k_docs, v_docs, q, k, K, V = request(b)
        tin = q.shape[0]
        n_rows = min(Tq, ORACLE_ROWS)
        rows = np.sort(rng.choice(Tq, size=n_rows, replace=False)) + (tin - Tq)
        pick = np.sort(rng.choice(len(docs), size=min(len(docs), ORACLE_DOCS), replace=False)) \
            if docs else np.zeros(0, np.int64)
        t0 = time.perf_counter()
        lay = O.compose_layout(lens, base, docs, int(wl.prefix_len[b]), Tq,
                               wl.block_table[b].numpy(), spec.page_size,
                               span_len=wl.meta["spans"][b])
        t1 = time.perf_counter()
        sub = dataclasses.replace(lay, doc_ids=[docs[i] for i in pick],
                                  doc_offset=[lay.doc_offset[i] for i in pick])
        if len(pick):
            O.relocate_docs(sub, [k_docs[i] for i in pick], [v_docs[i] for i in pick], base,
                            theta)
        t2 = time.perf_counter()
        ip = lay.inline_pos
        O.rotary(k, ip[:, None], theta)
        q_rot = O.rotary(q, ip[:, None], theta)
        lead = tin - Tq     # prefix and span rows, over the keys they can see
        if lead:
            O.attention(q_rot[:lead], ip[:lead], K[:ip[lead - 1] + 1], V[:ip[lead - 1] + 1])
        t3 = time.perf_counter()
        O.attention(q_rot[rows], ip[rows], K, V)
        t4 = time.perf_counter()
        doc_tok = sum(int(lens[x]) for x in docs)
        sub_tok = sum(int(lens[docs[i]]) for i in pick)
        reloc = (t2 - t1) * doc_tok / sub_tok if sub_tok else 0.0
        per_pass.append((t1 - t0) + reloc + (t3 - t2) + (t4 - t3) * Tq / n_rows)
        if K.shape[0] < 50_000:
            b = (b + 1) % spec.batch   # short requests: cycle over the batch
    t_total = sum(per_pass)
    rate = len(per_pass) * full.query_len / (t_total * full.layers)
    return {"value": rate, "passes": len(per_pass), "seconds": t_total, "per_pass": per_pass}


def run_oracle_subprocess(workload, seconds, passes=0):
    cores = len(os.sched_getaffinity(0))
    env = dict(os.environ)
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
        env[k] = str(cores)
    env["CUDA_VISIBLE_DEVICES"] = ""
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--oracle-sample",
                        workload, "--oracle-seconds", str(seconds), "--oracle-passes",
                        str(passes)],
                       capture_output=True, text=True, env=env, timeout=1200)
    if r.returncode != 0:
        raise RuntimeError(f"oracle sample failed: {r.stderr[-2000:]}")
    d = json.loads(r.stdout.strip().splitlines()[-1])
    d["cores"] = cores
    return d


def sample_desc(workload):
    from paper_2607_28069_gb300.workloads import WORKLOADS, draw_structure
    s = WORKLOADS[workload]
    m = len(draw_structure(s).docs[0])
    docs = (f"{ORACLE_DOCS} seeded documents of {m} re-rotated (time scaled by the request's "
            f"document tokens over theirs)" if m > ORACLE_DOCS else "every document re-rotated")
    rows = (f"{ORACLE_ROWS} seeded query rows of {s.query_len} over the full stitched context "
            f"(time scaled by {s.query_len}/{ORACLE_ROWS})" if s.query_len > ORACLE_ROWS else
            f"all {s.query_len} query rows over the full stitched context")
    one = "request 0" if sum(draw_structure(s).need) / s.batch >= 50_000 else "one request"
    return (f"fp64 numpy oracle, {one} x one layer per pass: layout, {docs}, inline RoPE, "
            f"prefix rows over the prefix, {rows}; rate scaled to {s.layers} layer(s) per "
            f"request")


# --------------------------------------------------------------- GPU arm
def main_gpu(args, rank, world):
    import torch

    import paper_2607_28069_gb300 as pic
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    from paper_2607_28069_gb300.workloads import WORKLOADS, generate

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pic.load()
    spec = WORKLOADS[args.workload]
    import dataclasses
    spec1 = spec if spec.decode_steps <= 1 else dataclasses.replace(spec, decode_steps=1)
    wl = generate(spec1, device=dev, gen_device=GPU_GEN.get(args.workload, "cuda"))
    layer_table = None
    if args.layer_rope:  # alternate a local-attention base (1e4) with the workload's base
        half = spec.head_dim // 2
        i = torch.arange(half, dtype=torch.float64)
        rows = [torch.pow(torch.tensor(1e4 if l % 2 == 0 else spec.rope_base, dtype=torch.float64),
                          -2.0 * i / spec.head_dim) for l in range(spec.layers)]
        layer_table = torch.stack(rows).to(dev)
    path = CacheHitPath(wl, prefill_splits=args.prefill_splits, decode_splits=args.decode_splits,
                        layer_inv_freq=layer_table)
    from paper_2607_28069_gb300.workloads import draw_structure
    work = work_of(spec, draw_structure(spec))
    L = spec.layers
    geom = path.geom
    psplits = pic.pic_prefill_num_splits(geom, spec.batch, path.max_inline, path.max_ctx,
                                         path.prefill_splits)

    # warm-up run and device-side status
    path.ttft_pass()
    if wl.q_dec is not None:
        path.decode_pass(0)
    torch.cuda.synchronize()
    code, detail = pic.pic_device_status()
    if code:
        raise RuntimeError(f"device status {code} detail {detail}")

    # The TTFT pass as CUDA graph(s) with timing events at every call boundary:
    # one graph with external event nodes when torch supports them, else one
    # graph per call with events between the replays.
    # rows: the separate calls of the path; the pass (value): pic_link for the
    # layout, every layer's relocation and the first layer's append, then the
    # attention of every layer (and the append of the later ones)
    calls = [("compose", path.compose), ("relocate", path.relocate)]
    for layer in range(L):
        calls.append(("append", (lambda l=layer: path.append(l))))
        calls.append(("attend", (lambda l=layer: path.attend(l))))
    pass_calls = [("link", (lambda: path.link(0))), ("attend", (lambda: path.attend(0)))]
    for layer in range(1, L):
        pass_calls.append(("append", (lambda l=layer: path.append(l))))
        pass_calls.append(("attend", (lambda l=layer: path.attend(l))))
    stream = torch.cuda.current_stream()
    try:
        bounds = [torch.cuda.Event(enable_timing=True, external=True)
                  for _ in range(len(calls) + 1)]
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            bounds[0].record()
            for i, (_, fn) in enumerate(calls):
                fn()
                bounds[i + 1].record()
        graphs = [g]
        single = True
        # the pass as it runs in service: no event nodes between the calls
        ends = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
        g_pass = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_pass):
            ends[0].record()
            for _, fn in pass_calls:
                fn()
            ends[1].record()
        # the link call alone, cold (its own row)
        lends = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
        g_link = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_link):
            lends[0].record()
            path.link(0)
            lends[1].record()
    except (TypeError, RuntimeError):
        graphs = []
        for _, fn in calls:
            gi = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gi):
                fn()
            graphs.append(gi)
        single = False
    dec_graph = None
    if wl.q_dec is not None:
        dec_graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(dec_graph):
            path.decode_pass(0)
    torch.cuda.synchronize()

    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush = torch.empty(max(2 * l2, 256 << 20), dtype=torch.uint8, device=dev)
    sleep_cycles = int(2e9 * max(50e-6, 5e-6 * len(graphs)))

    def pass_step():
        """Flush L2, then one pass with no timing nodes inside; returns ms."""
        flush.zero_()
        torch.cuda._sleep(sleep_cycles)
        g_pass.replay()
        torch.cuda.synchronize()
        return ends[0].elapsed_time(ends[1])

    def link_step():
        """Flush L2, then pic_link alone; returns ms."""
        flush.zero_()
        torch.cuda._sleep(sleep_cycles)
        g_link.replay()
        torch.cuda.synchronize()
        return lends[0].elapsed_time(lends[1])

    def one_step():
        """Flush L2, then one pass; returns per-call ms after synchronising."""
        flush.zero_()
        torch.cuda._sleep(sleep_cycles)   # GPU busy while the host enqueues
        if single:
            graphs[0].replay()
            torch.cuda.synchronize()
            return [bounds[i].elapsed_time(bounds[i + 1]) for i in range(len(calls))]
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(len(graphs) + 1)]
        evs[0].record(stream)
        for i, gi in enumerate(graphs):
            gi.replay()
            evs[i + 1].record(stream)
        torch.cuda.synchronize()
        return [evs[i].elapsed_time(evs[i + 1]) for i in range(len(calls))]

    W, K = args.warmup, args.steps
    torch.cuda._sleep(int(2e9 * 0.3))   # let the clocks ramp before warm-up
    for _ in range(W):
        if single:
            pass_step()
            link_step()
        one_step()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    per_call, pass_ms, link_ms = [], [], []
    with ClockSampler(dev) as clk:
        for _ in range(K):
            if single:
                pass_ms.append(pass_step())
                link_ms.append(link_step())
            per_call.append(one_step())
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    # value: the pass as served (no timing nodes between calls) when torch
    # supports event nodes in graphs; else the per-call graphs' sum
    step_ms = pass_ms if single else [sum(x) for x in per_call]
    phase_ms = {}
    for x in per_call:
        for (name, _), ms in zip(calls, x):
            phase_ms.setdefault(name, []).append(ms)
    total_ms = max_over_ranks(sum(step_ms), world, dev)
    ms_per_step = total_ms / K
    value = job_rate(work["query_tokens"], K, world, total_ms)

    # per-row averages over the timed steps (ms per step)
    per_step = {name: sum(v) / K for name, v in phase_ms.items()}
    peaks, peak_src = load_peaks()
    rows = {
        "a1_compose": {"ms": per_step["compose"], "launches": 1},
        "a2_a3_relocate": {
            "ms": per_step["relocate"], "launches": 1,
            "bytes": work["relocate_bytes"],
            "gbs": work["relocate_bytes"] / (per_step["relocate"] * 1e6)},
        "a4_append": {"ms": per_step["append"], "launches": L,
                      "bytes": work["append_bytes"],
                      "gbs": work["append_bytes"] / (per_step["append"] * 1e6)},
        "a5_attend": {"ms": per_step["attend"], "launches": L * (2 if psplits > 1 else 1),
                      "flops": work["attend_flops"], "splits": psplits,
                      "tflops": work["attend_flops"] / (per_step["attend"] * 1e9)},
    }
    rows["a2_a3_relocate"]["frac_hbm"] = rows["a2_a3_relocate"]["gbs"] / peaks["hbm_gbs"]
    if link_ms:
        lms = sum(link_ms) / len(link_ms)
        link_bytes = work["relocate_bytes"] + work["append_bytes"] / L
        rows["a1_a4_link"] = {
            "ms": lms, "launches": 1, "bytes": link_bytes, "gbs": link_bytes / (lms * 1e6),
            "frac_hbm": link_bytes / (lms * 1e6) / peaks["hbm_gbs"],
            "note": "pic_link: layout, every layer's relocation and layer 0's inline append in "
                    "one launch (what the pass runs); rows a1-a4 time the separate calls"}
    rows["a5_attend"]["frac_bf16"] = rows["a5_attend"]["tflops"] / peaks["bf16_tflops"]
    # kernels of the timed pass: pic_link, the later layers' appends, attention (+ merge)
    launches = (1 + (L - 1) + rows["a5_attend"]["launches"]) if single else \
        (1 + 1 + L + rows["a5_attend"]["launches"])

    # decode (outside the TTFT boundary), same run
    if dec_graph is not None:
        dsplits = pic.pic_decode_num_splits(geom, spec.batch, path.max_ctx, args.decode_splits)
        dts = []
        for k in range(max(3, K // 2) + 2):
            flush.zero_()
            torch.cuda._sleep(sleep_cycles)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            dec_graph.replay()
            e1.record(stream)
            torch.cuda.synchronize()
            if k >= 2:
                dts.append(e0.elapsed_time(e1))
        dms = sum(dts) / len(dts)
        rows["a6_decode"] = {
            "ms": dms, "launches": L * (3 if dsplits > 1 else 2), "splits": dsplits,
            "bytes": work["decode_bytes"], "gbs": work["decode_bytes"] / (dms * 1e6),
            "tok_s": spec.batch / (dms / 1e3)}
        rows["a6_decode"]["frac_hbm"] = rows["a6_decode"]["gbs"] / peaks["hbm_gbs"]

    # fused rotate-on-load pass (a7): compose, then per layer append + fused
    # attention reading the documents from the pool; no relocation
    if args.fused or args.workload == "stress_128k_b4":
        fcalls = [("compose", path.compose)]
        for layer in range(L):
            fcalls.append(("append", (lambda l=layer: path.append(l))))
            fcalls.append(("fused", (lambda l=layer: path.attend_fused(l))))
        fb = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(len(fcalls) + 1)]
        fg = torch.cuda.CUDAGraph()
        with torch.cuda.graph(fg):
            fb[0].record()
            for i, (_, fn) in enumerate(fcalls):
                fn()
                fb[i + 1].record()
        torch.cuda.synchronize()
        f_tot, f_att = [], []
        for k in range(W + max(2, K)):
            flush.zero_()
            torch.cuda._sleep(sleep_cycles)
            fg.replay()
            torch.cuda.synchronize()
            ms = [fb[i].elapsed_time(fb[i + 1]) for i in range(len(fcalls))]
            if k >= W:
                f_tot.append(sum(ms))
                f_att.append(sum(x for (nm, _), x in zip(fcalls, ms) if nm == "fused"))
        fms, fatt = sum(f_tot) / len(f_tot), sum(f_att) / len(f_att)
        rows["a7_fused"] = {
            "ms": fms, "attend_ms": fatt, "launches": 1 + L + L * (2 if psplits > 1 else 1),
            "flops": work["attend_flops"], "tflops": work["attend_flops"] / (fatt * 1e9),
            "frac_bf16": work["attend_flops"] / (fatt * 1e9) / peaks["bf16_tflops"],
            "query_tok_s": work["query_tokens"] / (fms / 1e3),
            "speedup_vs_materialised": ms_per_step / fms}

    # launch floor of the pass: empty programmatic-dependent kernels with the
    # pass's launch shapes (link, then per layer the attention and its merge,
    # and for later layers the append first), timed like the pass
    if args.floor:
        B, Hkv, d = spec.batch, spec.kv_heads, spec.head_dim
        G = spec.q_heads // Hkv
        m_tiles = -(-path.max_inline * G // 128)
        pairs = -(-m_tiles // 2)
        tile = 128 * d * 2
        attn_smem = 2 * tile + 3 * tile + 2 * tile + 256 + 3 * 8 * 8 + 1024
        tok = 16 if Hkv * d >= 1024 else 32
        shapes = [((-(-path.max_ctx // tok), B, 1), 256, 0)]
        for layer in range(L):
            if layer > 0:
                shapes.append(((max(path.max_inline, -(-m_tiles * 128 // G)), B, 1), 256, 0))
            shapes.append(((pairs * psplits, Hkv, B), 384, attn_smem))
            if psplits > 1:
                u = 2 if psplits <= 2 else (4 if psplits <= 4 else 8)
                rows_m = B * Hkv * m_tiles * 128
                shapes.append(((-(-rows_m // (8 * (8 // u))), 1, 1), 256, 0))
        fe = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
        gf = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gf):
            fe[0].record()
            pic.pic_launch_probe(shapes)
            fe[1].record()
        torch.cuda.synchronize()
        fts = []
        for k in range(W + max(3, K)):
            flush.zero_()
            torch.cuda._sleep(sleep_cycles)
            gf.replay()
            torch.cuda.synchronize()
            if k >= W:
                fts.append(fe[0].elapsed_time(fe[1]))
        fl_ms = sum(fts) / len(fts)
        rows["floor"] = {"ms": fl_ms, "launches": len(shapes), "frac_of_pass": fl_ms / ms_per_step,
                         "note": "empty programmatic-dependent kernels with the pass's launch "
                                 "shapes (grid, block, dynamic shared memory), one graph, "
                                 "timed like the pass"}

    # attention-deviation diagnostic (off the serving path): D_r between the
    # relocated cache and the documents copied without re-rotation, layer 0
    if args.deviation:
        pathB = CacheHitPath(wl, prefill_splits=args.prefill_splits)
        pathB.compose()
        pic.pic_relocate_mapped(pathB.geom, wl.k_pool, wl.v_pool, pathB.tok_map,
                         torch.zeros_like(pathB.doc_delta), pathB.slot_mapping, wl.num_pages,
                         pathB.k_cache, pathB.v_cache, 0, 1)
        pathA = CacheHitPath(wl, prefill_splits=args.prefill_splits, with_lse=True)
        pathA.compose()
        pathA.relocate(0, 1)
        pathB.lse = torch.empty_like(pathA.lse)
        for pth in (pathA, pathB):
            pth.append(0)
            pic.pic_attend_prefill(pth.geom, 0, pth.inline_pos, wl.inline_len, pth.max_ctx,
                                   wl.block_table, wl.num_pages, pth.k_cache, pth.v_cache,
                                   pth.out[0], pth.lse[0], pth.prefill_splits, pth.ws_prefill)
        qlen = torch.full((spec.batch,), spec.query_len, dtype=torch.int32, device=dev)
        dsum = torch.empty((spec.batch, 2), dtype=torch.float64, device=dev)
        dcnt = torch.empty((spec.batch, 2), dtype=torch.int64, device=dev)

        def dev_call():
            pic.pic_attention_deviation(pathA.geom, 0, pathA.inline_pos, wl.inline_len, qlen,
                                        wl.req_doc_ids, wl.doc_len, pathA.doc_offset,
                                        pathA.slot_mapping, wl.num_pages,
                                        pathA.k_cache, pathB.k_cache, pathA.lse[0], pathB.lse[0],
                                        pathA.ws_prefill, dsum, dcnt, (0.0, 0.1, 0.9),
                                        max_query_len=spec.query_len)
        dts = []
        for k in range(W + max(3, K // 2)):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            dev_call()
            e1.record(stream)
            torch.cuda.synchronize()
            if k >= W:
                dts.append(e0.elapsed_time(e1))
        dv_ms = sum(dts) / len(dts)
        terms = int(dcnt.sum().item())          # (row, head, key) terms in the regions
        flops = 2 * 2 * spec.head_dim * terms   # two dot products (QK^T of A and of B) per term
        d_r = (dsum.sum(0) / dcnt.sum(0).clamp(min=1)).tolist()
        rows["next4_deviation"] = {
            "ms": dv_ms, "launches": 1, "terms": terms, "tflops": flops / (dv_ms * 1e9),
            "frac_bf16": flops / (dv_ms * 1e9) / peaks["bf16_tflops"], "D_pre": d_r[0],
            "D_int": d_r[1],
            "note": "layer 0: relocated cache vs documents copied without re-rotation; FLOPs "
                    "count the region terms only (two 2-d dot products each)"}
        del pathA, pathB

    # dominant kernel of the step -> roofline object: attention, or the data
    # movement the pass runs (pic_link when the pass is one graph, else relocate)
    move_ms = rows["a1_a4_link"]["ms"] if "a1_a4_link" in rows else per_step["relocate"]
    if per_step["attend"] >= move_ms:
        per_launch_ms = per_step["attend"] / L
        flops_launch = work["attend_flops"] / L
        achieved = flops_launch / (per_launch_ms * 1e9)
        traffic = ncu_traffic(f"attn_kernel|{args.workload}", "pic_prefill.cu")
        roof = {"kernel": "attn_kernel (pic_attend_prefill)", "bound": "tensor",
                "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                "frac": achieved / peaks["bf16_tflops"], "traffic": traffic,
                "peak_source": f"{peak_src} bf16 burst"}
        # A kernel timed inside a long step (a second or more of back-to-back
        # steps, under the power cap) also against the sustained matmul rate;
        # `peak` stays the burst figure, the stricter of the two.
        if K * ms_per_step >= 1000.0 and peaks.get("bf16_tflops_sustained"):
            roof["peak_sustained"] = peaks["bf16_tflops_sustained"]
            roof["frac_sustained"] = achieved / peaks["bf16_tflops_sustained"]
    elif "a1_a4_link" in rows:
        achieved = rows["a1_a4_link"]["gbs"]
        traffic = ncu_traffic(f"link_kernel|{args.workload}", "pic_link.cu")
        roof = {"kernel": "link_kernel (pic_link)", "bound": "hbm",
                "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / peaks["hbm_gbs"], "traffic": traffic,
                "peak_source": f"{peak_src} copy"}
    else:
        achieved = rows["a2_a3_relocate"]["gbs"]
        traffic = ncu_traffic(f"relocate_kernel|{args.workload}", "pic_relocate.cu")
        roof = {"kernel": "relocate_kernel (pic_relocate)", "bound": "hbm",
                "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / peaks["hbm_gbs"], "traffic": traffic,
                "peak_source": f"{peak_src} copy"}

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        # Per-request inputs packed into one pinned host buffer (pipeline
        # API): every step copies the whole request in and every layer's
        # attention output back out, overlapped with the compute
        # (CacheHitPath.served_pass: the per-request fields and layer 0's
        # projections by the library's copy kernel, later layers' inputs and
        # earlier layers' outputs on two copy-engine streams, the last
        # layer's output by the copy kernel), captured as one graph that
        # reads and writes the same host buffers on every replay.
        host_req = path.pack_request_inputs()
        host_out = torch.empty(path.out.shape, dtype=path.out.dtype, pin_memory=True)
        h2d = host_req.numel()
        d2h = host_out.numel() * host_out.element_size()
        up_stream, down_stream = torch.cuda.Stream(), torch.cuda.Stream()
        g2 = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g2):
            path.served_pass(host_req, host_out, up_stream, down_stream)
        torch.cuda.synchronize()
        e_ms = []
        for k in range(W + K):
            flush.zero_()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            g2.replay()
            e1.record(stream)
            torch.cuda.synchronize()
            if k >= W:
                e_ms.append(e0.elapsed_time(e1))
        e_total = max_over_ranks(sum(e_ms), world, dev)
        e2e = {"value": job_rate(work["query_tokens"], K, world, e_total),
               "unit": "query_tokens/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}

    code, detail = pic.pic_device_status()
    if code:
        raise RuntimeError(f"device status {code} detail {detail} after the timed run")

    config = bench_config(args.workload, world)
    if not single:
        config["timing"] = "one CUDA graph per call, events between replays"
    out = {
        "metric": METRIC,
        "value": value, "unit": "query_tokens/s", "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": config,
        "gpu_launches": launches,
        "rows": rows,
        "rows_ms_per_step": sum(per_step.values()),  # the row graph, with its event nodes
        "roofline": roof,
        "clocks": clk.summary(),
        "e2e": e2e,
    }
    return out


def main_reference(args):
    """The reference arm: the CPU oracle on the machine's host cores, W untimed
    and K timed passes (one subprocess, the workload generated once), each a
    bounded sample of the workload (see oracle_sample)."""
    cores = len(os.sched_getaffinity(0))
    W, K = args.warmup, args.steps
    d = run_oracle_subprocess(args.workload, 0.0, passes=W + K)
    timed = d["per_pass"][W:]
    from paper_2607_28069_gb300.workloads import WORKLOADS
    spec = WORKLOADS[args.workload]
    value = len(timed) * spec.query_len / (sum(timed) * spec.layers)
    return {
        "impl": "reference", "metric": METRIC, "value": value,
        "unit": "query_tokens/s", "n_gpus": args.gpus, "steps": K,
        "warmup": W, "ms_per_step": 1e3 * spec.batch * spec.query_len / value,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": bench_config(args.workload, args.gpus),
        "cpu_baseline": {"value": value, "unit": "query_tokens/s", "cores": cores,
                         "kind": "oracle",
                         "sample": sample_desc(args.workload) +
                         f"; {K} timed passes after {W} untimed, one per step"},
        "e2e": {"value": value, "unit": "query_tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def main(argv=None):
    args = parse_args(argv)
    if args.oracle_sample:
        print(json.dumps(oracle_sample(args.oracle_sample, args.oracle_seconds,
                                       args.oracle_passes)))
        return 0
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank != 0:
            return 0
        print(json.dumps(main_reference(args)))
        return 0
    import torch
    if world > 1:
        torch.distributed.init_process_group("nccl")
    # the oracle baseline runs before the GPU work so its subprocess starts clean
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        d = run_oracle_subprocess(args.workload, args.oracle_seconds)
        cpu = {"value": d["value"], "unit": "query_tokens/s", "cores": d["cores"],
               "kind": "oracle", "sample": sample_desc(args.workload) +
               f"; {d['passes']} passes in {d['seconds']:.1f} s"}
    out = main_gpu(args, rank, world)
    out["cpu_baseline"] = cpu
    if rank == 0:
        print(json.dumps(out))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
