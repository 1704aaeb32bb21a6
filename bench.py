#!/usr/bin/env python
"""Tree-verify benchmark: verify steps/s at the 7B shape (KV 2400, 64-node
tree) and the HBM roofline of the attention kernel.

One step = 6 draft-layer expansions (width 8) over 65536-entry draft rows,
the top-63 rerank, tree attention over all 32 layers (32 heads x 128, prefix
2400), the acceptance walk and the KV commit of the accepted path: every row
of the hot path, as one CUDA graph of library launches.  The attention
kernel's time per launch (the roofline) comes from a second timed region in
the same run: the 32 attention layers alone, back to back as in the step.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 7b|llamagen|c1|c4]
                  [--mode greedy|spec_det] [--impl adt|reference]

Prints one JSON line.  With torchrun (N > 1) every rank runs an independent
replica on its own GPU (the path has no cross-GPU exchange) and rank 0
reports the whole-job throughput (weak scaling).
"""
from __future__ import annotations

import argparse
import datetime as _dt
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

WORKLOADS = {
    "7b": dict(name="7B-class (Anole / Lumina-mGPT shape) tree verify: 32 layers, 32 heads x 128, KV 2400, "
                    "64-node tree (depth 6, width 8), vocab 65536, batch 1",
               layers=32, H=32, Hkv=32, D=128, V=65536, kv_len=[2400], depth=[6], width=[8], max_nodes=64),
    "llamagen": dict(name="LlamaGen-XL-shaped tree verify: 36 layers, 20 heads x 64, KV 696 (120 text + 576 image), "
                          "64-node tree (depth 6, width 8), vocab 16384, batch 1",
                     layers=36, H=20, Hkv=20, D=64, V=16384, kv_len=[696], depth=[6], width=[8], max_nodes=64),
    "c1": dict(name="single verify step: 1 layer, 8 heads x 64, KV 512, 26-node tree (depth 4, width 4), "
                    "vocab 16384, batch 1",
               layers=1, H=8, Hkv=8, D=64, V=16384, kv_len=[512], depth=[4], width=[4], max_nodes=26),
    # prefix lengths ~ U{600..2400}, depths ~ U{2..10}, widths ~ U{1..8} (numpy default_rng(20251221), in
    # that order): one batched step of the adjacency-adaptive sweep, each image's tree its own shape
    "c4": dict(name="adjacency-adaptive ragged batch: 8 images at the 7B shape (32 layers, 32 heads x 128, "
                    "vocab 65536), KV 600-2400, per-image depth 2-10 and width 1-8, trees of up to 64 nodes",
               layers=32, H=32, Hkv=32, D=128, V=65536, kv_len=[751, 1596, 1444, 640, 1427, 1245, 2352, 1248],
               depth=[4, 7, 8, 7, 6, 6, 7, 6], width=[6, 8, 4, 2, 2, 1, 6, 4], max_nodes=64),
}

# DRAM bytes (read + write) of one tree_attn launch at the 7B shape, from one
# ncu capture; valid only for the kernel source with this SHA-256 prefix.
HOST_MARKER = b"// ---------------------------------------------------------------- host side"
NCU_TRAFFIC = {
    # dram__bytes_read.sum + dram__bytes_write.sum = 41,496,064 + 0
    "53c1a5e07c7c7659": 41496064,
}


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def max_over_ranks(x: float, world: int) -> float:
    """The largest of every rank's x (the slowest replica sets the job's
    time); x itself with one rank."""
    if world <= 1:
        return x
    import torch
    dev = "cuda" if torch.distributed.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def job_throughput(ms_per_step: float, world: int) -> float:
    """Whole-job steps/s: every rank verifies its own replica's step (weak
    scaling), in the slowest rank's time."""
    return world * 1e3 / ms_per_step


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def attn_source_sha():
    """SHA-256 prefix of the attention kernel's device code: tree_attn.cu up to
    its host-side section (host-only edits do not change the kernel)."""
    with open(os.path.join(ROOT, "paper_2512_21857_gb300", "csrc", "tree_attn.cu"), "rb") as f:
        src = f.read()
    cut = src.find(HOST_MARKER)
    return hashlib.sha256(src if cut < 0 else src[:cut]).hexdigest()[:16]


# ------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "100", "-i", str(self.dev)], stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self, t0, t1):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            try:
                ts = _dt.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                rows.append((ts, float(parts[2]), float(parts[3]), parts[6:10]))
            except ValueError:
                continue
        inside = [r for r in rows if t0 - 0.05 <= r[0] <= t1 + 0.05]
        use = inside or rows
        if not use:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        reasons = sorted({n for r in use for n, v in zip(self.NAMES, r[3]) if v.lower().startswith("active")})
        return {"sm_mhz": statistics.median(r[1] for r in use), "sm_max_mhz": max(r[2] for r in use),
                "reasons": reasons, "samples": len(use), "samples_in_timed_region": len(inside)}


class NvmlSampler:
    """SM clock and clock-event reasons read through NVML (ctypes on the
    driver's libnvidia-ml) every ~1 ms in a thread, so that a timed region of
    a few milliseconds still holds samples.  Reads only."""
    REASONS = {0x8: "hw_slowdown", 0x40: "hw_thermal_slowdown", 0x20: "sw_thermal_slowdown", 0x4: "sw_power_cap"}

    def __init__(self, device_index):
        import ctypes
        import threading
        self.ok = False
        self.samples = []
        self._stop = threading.Event()
        try:
            self.lib = ctypes.CDLL("libnvidia-ml.so.1")
            if self.lib.nvmlInit_v2() != 0:
                return
            self.h = ctypes.c_void_p()
            if self.lib.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(device_index), ctypes.byref(self.h)) != 0:
                return
            self.max_mhz = ctypes.c_uint(0)
            self.lib.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(self.max_mhz))  # NVML_CLOCK_SM
            self.ok = True
        except OSError:
            return
        self.thread = threading.Thread(target=self._run, daemon=True)

    def _run(self):
        import ctypes
        mhz = ctypes.c_uint(0)
        reasons = ctypes.c_ulonglong(0)
        get_reasons = getattr(self.lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            self.lib.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self._stop.is_set():
            if self.lib.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(mhz)) == 0 and \
                    get_reasons(self.h, ctypes.byref(reasons)) == 0:
                self.samples.append((time.time(), mhz.value, reasons.value))
            time.sleep(0.001)

    def start(self):
        if self.ok:
            self.thread.start()

    def stop(self, t0, t1):
        if not self.ok:
            return None
        self._stop.set()
        self.thread.join(timeout=2)
        inside = [r for r in self.samples if t0 <= r[0] <= t1]
        use = inside or self.samples
        if not use:
            return None
        bits = 0
        for r in use:
            bits |= r[2]
        return {"sm_mhz": statistics.median(r[1] for r in use), "sm_max_mhz": self.max_mhz.value,
                "reasons": sorted(n for m, n in self.REASONS.items() if bits & m), "samples": len(use),
                "samples_in_timed_region": len(inside), "source": "nvml, 1 ms"}


# ------------------------------------------------------------------ GPU arm

def fill_inputs_on_device(step, seed):
    """Seeded synthetic inputs drawn on the device (bf16 ~ N(0,1) caches and
    projections, fp32 ~ N(0, 3^2) logits, 24-bit uniforms)."""
    import torch
    g = torch.Generator(device=step.device)
    g.manual_seed(seed)

    def normal_(t, std=1.0):
        t.copy_((torch.randn(t.shape, generator=g, device=step.device) * std).to(t.dtype))

    for name in ("k_cache", "v_cache", "q", "k_tree", "v_tree"):
        normal_(getattr(step, name))
    for rows in step.draft_rows:
        normal_(rows, 3.0)
    normal_(step.target, 3.0)
    for t in (step.u_accept, step.u_sample):
        t.copy_(torch.randint(0, 1 << 24, t.shape, generator=g, device=step.device).float() * 2.0 ** -24)
    step.root_token.copy_(torch.randint(0, step.shape.V, step.root_token.shape, generator=g, device=step.device))


def run_gpu(args, wl, rank, world):
    import torch
    from paper_2512_21857_gb300 import binding as B
    from paper_2512_21857_gb300 import build as libbuild
    from paper_2512_21857_gb300.verify_step import StepShape, TreeVerifyStep

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    libbuild.build()
    B.lib()
    mode = {"greedy": B.ACCEPT_GREEDY, "spec_det": B.ACCEPT_SPEC_DET}[args.mode]
    shape = StepShape(layers=wl["layers"], H=wl["H"], Hkv=wl["Hkv"], D=wl["D"], V=wl["V"], kv_len=wl["kv_len"],
                      depth=wl["depth"], width=wl["width"], max_nodes=wl["max_nodes"], mode=mode, temperature=1.0)
    step = TreeVerifyStep(shape, input_slots=2)
    fill_inputs_on_device(step, 20251221 + rank)
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    # eager pass first (per-device one-time set-up happens outside capture)
    with torch.cuda.stream(stream):
        step.launch(stream)
    torch.cuda.synchronize()
    if B.adt_get_device_error(stream) != 0:
        raise RuntimeError("device error flag set during the eager pass")
    # The step is one CUDA graph (its kernels chained by programmatic
    # dependent launch, no host work between them).  The attention layers
    # are also captured alone, back to back as inside the step, to time the
    # attention kernel for the roofline in a second timed region.
    step_graph = torch.cuda.CUDAGraph()
    attn_graph = torch.cuda.CUDAGraph()
    # The draft-tree expansion calls of image 0 (depth calls, F = 1 then the
    # width), back to back as inside the step, timed alone after the others.
    expand_graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(step_graph, stream=stream):
            step.launch(stream)
        with torch.cuda.graph(attn_graph, stream=stream):
            for layer in range(shape.layers):
                step.launch_attention(layer, stream)
        with torch.cuda.graph(expand_graph, stream=stream):
            step.launch_draft_image(0, stream, rerank=False)
    torch.cuda.synchronize()

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step_graph.replay()
            attn_graph.replay()
            expand_graph.replay()
    torch.cuda.synchronize()

    K = args.steps
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ea0, ea1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ee0, ee1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    sampler.start()
    nvml = NvmlSampler(local)
    nvml.start()
    time.sleep(0.4)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    t0 = time.time()
    step_ev = [torch.cuda.Event(enable_timing=True) for _ in range(K + 1)]
    with torch.cuda.stream(stream):
        ev0.record(stream)
        step_ev[0].record(stream)
        for i in range(K):
            step_graph.replay()
            step_ev[i + 1].record(stream)
        ev1.record(stream)
        ea0.record(stream)
        for _ in range(K):
            attn_graph.replay()
        ea1.record(stream)
        ee0.record(stream)
        for _ in range(K):
            expand_graph.replay()
        ee1.record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    if world > 1:
        torch.distributed.barrier()
    clocks = sampler.stop(t0, t1)
    fine = nvml.stop(t0, t1)
    if fine is not None:
        fine["nvidia_smi"] = clocks
        clocks = fine
    step_ms = ev0.elapsed_time(ev1) / K
    per_step = sorted(step_ev[i].elapsed_time(step_ev[i + 1]) for i in range(K))
    pct = {f"p{q}": per_step[min(K - 1, int(round(q / 100 * (K - 1))))] for q in (10, 50, 90)}
    attn_ms = ea0.elapsed_time(ea1) / (K * shape.layers)
    expand_calls = int(shape.depth[0])
    expand_us = ee0.elapsed_time(ee1) * 1000.0 / (K * expand_calls)
    errbits = B.adt_get_device_error(stream)
    if errbits:
        raise RuntimeError(f"device error bits {errbits:#x} during the timed steps")
    step_ms = max_over_ranks(step_ms, world)

    # End to end through the public API: every step copies its inputs from
    # pinned host memory into one of two input slots and reads its result
    # back; the copy of step i + 1 (its own stream) overlaps the compute of
    # step i, as a serving loop would run it.
    step.use_slot(1)
    for name in step.STEP_INPUTS:
        src = getattr(step, "_slots")[0][name]
        dst = getattr(step, name)
        if isinstance(src, list):
            for a, b_ in zip(dst, src):
                a.copy_(b_)
        else:
            dst.copy_(src)
    step_graph1 = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(step_graph1, stream=stream):
            step.launch(stream)
    step.use_slot(0)
    torch.cuda.synchronize()
    slot_graphs = [step_graph, step_graph1]
    slot_inputs = []
    for i in range(2):
        step.use_slot(i)
        slot_inputs.append(step.step_input_tensors())
    step.use_slot(0)
    host_in = [t.cpu().pin_memory() for t in slot_inputs[0]]
    outputs = [step.path, step.accept_len, step.bonus, step.kv_len_out]
    host_out = [[torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in outputs] for _ in range(2)]
    h2d = sum(t.numel() * t.element_size() for t in host_in)
    d2h = sum(t.numel() * t.element_size() for t in host_out[0])
    copy_stream = torch.cuda.Stream()
    copied = [torch.cuda.Event() for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]
    done = [torch.cuda.Event() for _ in range(2)]

    def issue(i):
        sl = i % 2
        if i >= 2:
            copy_stream.wait_event(consumed[sl])
        with torch.cuda.stream(copy_stream):
            for d, h in zip(slot_inputs[sl], host_in):
                d.copy_(h, non_blocking=True)
            copied[sl].record(copy_stream)
        stream.wait_event(copied[sl])
        with torch.cuda.stream(stream):
            slot_graphs[sl].replay()
            consumed[sl].record(stream)
            for h, d in zip(host_out[sl], outputs):
                h.copy_(d, non_blocking=True)
            done[sl].record(stream)

    K2 = max(3, min(K, args.e2e_steps))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    copy_stream.wait_event(e0)
    issue(0)
    for i in range(K2):
        if i + 1 < K2:
            issue(i + 1)
        done[i % 2].synchronize()
        _ = int(host_out[i % 2][1][0])  # the host reads step i's result
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1) / K2
    e2e_ms = max_over_ranks(e2e_ms, world)

    ab = step.algorithmic_bytes()
    peak, peak_kind = measured_peaks()
    achieved = ab["attention_per_layer"] / (attn_ms * 1e-3) / 1e9
    sha = attn_source_sha()
    traffic = NCU_TRAFFIC.get(sha) if args.workload == "7b" else None
    return dict(step_ms=step_ms, step_pct=pct, attn_ms=attn_ms, clocks=clocks, e2e_ms=e2e_ms, h2d=h2d, d2h=d2h,
                launches=K * (step.kernel_launches_per_step() + shape.layers + expand_calls), achieved=achieved,
                peak=peak, peak_kind=peak_kind, expand_us=expand_us, expand_calls=expand_calls,
                traffic=traffic, attn_bytes=ab["attention_per_layer"], step_bytes=ab["attention"], sha=sha)


# ------------------------------------------------------------------ oracle (CPU) samples

class OracleSample:
    """A bounded sample of one verify step run by the oracle, extrapolated to
    the full step: `heads` query heads of `layers_sampled` layers of
    attention (all tree nodes), `rows_sampled` draft rows of expansion, the
    full rerank and greedy acceptance walk, and the KV commit of one layer.
    Inputs are drawn once; run() times only the oracle calls."""

    def __init__(self, wl, seed, heads, layers_sampled, rows_sampled, image=0, nodes_sampled=0):
        import numpy as np

        from paper_2512_21857_gb300 import synth

        self.wl = wl
        self.image = image
        H, Hkv, D, V, L = wl["H"], wl["Hkv"], wl["D"], wl["V"], wl["kv_len"][image]
        k, depth, nmax = wl["width"][image], wl["depth"][image], wl["max_nodes"]
        self.n = n = min(nmax, k + (depth - 1) * k * k + 1)
        # attention over the first nq nodes (parents precede children, so a
        # prefix of the node list is itself a tree), extrapolated to n
        self.nq = nq = n if nodes_sampled <= 0 else max(1, min(n, nodes_sampled))
        self.hs = hs = max(1, min(heads, H))
        self.layers_sampled = layers_sampled
        self.rows_sampled = rows_sampled
        self.total_rows = 1 + (depth - 1) * k
        g = synth.rng(seed, "oracle_sample")
        self.tb = synth.tree_batch([n], V, seed)
        self.q = synth.bf16_normal((n, hs, D), seed, "q").double().numpy()
        self.kc = synth.bf16_normal((1, hs, L, D), seed, "kc").double().numpy()
        self.vc = synth.bf16_normal((1, hs, L, D), seed, "vc").double().numpy()
        self.kt = synth.bf16_normal((n, hs, D), seed, "kt").double().numpy()
        self.vt = synth.bf16_normal((n, hs, D), seed, "vt").double().numpy()
        self.rows_sampled = rows_sampled = min(rows_sampled, self.total_rows)
        self.rows = synth.f32_normal((rows_sampled, V), seed, "rows")
        self.target = synth.f32_normal((n, V), seed, "target")
        C = k + (depth - 1) * k * k
        self.cand_tok = g.integers(0, V, size=C).astype(np.int32)
        self.cand_score = -np.sort(g.random(C)).astype(np.float32)
        self.cand_par = -np.ones(C, np.int32)
        self.kc16 = np.zeros((1, 1, Hkv, L + nmax, D), np.int16)
        self.kt16 = np.zeros((1, n, Hkv, D), np.int16)
        self.desc = (f"oracle (numpy fp64, 1 thread) on {hs} of {H} heads x {layers_sampled} of {wl['layers']} "
                     f"layers of attention" + (f" for {nq} of {n} tree nodes" if nq < n else "") +
                     f", {rows_sampled} of {self.total_rows} draft rows of expansion, full "
                     f"rerank and greedy walk, 1 of {wl['layers']} layers of KV commit; extrapolated linearly "
                     f"to one full step")

    def run(self):
        import numpy as np

        import oracle

        wl = self.wl
        L, D, n, k = wl["kv_len"][self.image], wl["D"], self.n, wl["width"][self.image]
        t = t_start = time.perf_counter()
        nq = self.nq
        for _ in range(self.layers_sampled):
            oracle.tree_attention(self.q[:nq], self.kc, self.vc, [L], self.kt[:nq], self.vt[:nq],
                                  self.tb.parents[:nq], [0, nq], 1.0 / math.sqrt(D))
        t_attn = ((time.perf_counter() - t) / self.layers_sampled * wl["layers"] * (wl["H"] / self.hs)
                  * (n / nq))
        t = time.perf_counter()
        oracle.tree_expand(self.rows, np.zeros(self.rows_sampled, np.float32), k, k)
        t_exp = (time.perf_counter() - t) / self.rows_sampled * self.total_rows
        t = time.perf_counter()
        oracle.tree_rerank(self.cand_tok, self.cand_score, self.cand_par, 1, n)
        oracle.tree_accept(self.target, None, self.tb.tokens, self.tb.parents, [0, n], oracle.ACCEPT_GREEDY)
        t_acc = time.perf_counter() - t
        t = time.perf_counter()
        oracle.kv_compact(self.kc16, self.kc16, [L], self.kt16, self.kt16, [0, n], [[0, 1]])
        t_cmp = (time.perf_counter() - t) * wl["layers"]
        self.wall = time.perf_counter() - t_start   # the seconds actually spent
        self.parts = dict(attn=t_attn, expand=t_exp, accept=t_acc, commit=t_cmp)
        return t_attn + t_exp + t_acc + t_cmp

    def run_attention_only(self):
        """One sampled layer of attention for this sample's heads (seconds)."""
        wl = self.wl
        nq = self.nq
        t = time.perf_counter()
        oracle_mod().tree_attention(self.q[:nq], self.kc, self.vc, [wl["kv_len"][self.image]], self.kt[:nq],
                                    self.vt[:nq], self.tb.parents[:nq], [0, nq], 1.0 / math.sqrt(wl["D"]))
        return time.perf_counter() - t


def oracle_mod():
    import oracle
    return oracle


def _attention_worker(job):
    """All-core leg: one worker process builds a sample of `heads` heads and
    times one layer of the oracle's attention for them (single-threaded)."""
    wl_key, seed, heads, image = job
    smp = OracleSample(WORKLOADS[wl_key], seed, heads, 1, 1, image=image)
    smp.run_attention_only()  # first touch of the inputs, untimed
    return smp.run_attention_only()


def cpu_model():
    """The host CPU's model name (lscpu), for the record."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    import platform
    return platform.processor() or platform.machine()


def cpu_sample_subprocess(wl_key, heads, layers_sampled, rows_sampled, reps, nodes=0, procs=1):
    """Runs oracle samples in a fresh single-threaded process (and, with
    procs > 1, the all-core attention leg in a pool of that many)."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    cmd = [sys.executable, os.path.abspath(__file__), "--cpu-sample", wl_key, "--cpu-heads", str(heads),
           "--cpu-layers", str(layers_sampled), "--cpu-rows", str(rows_sampled), "--cpu-reps", str(reps),
           "--cpu-nodes", str(nodes), "--cpu-procs", str(procs)]
    out = subprocess.run(cmd, capture_output=True, text=True, env=env, timeout=1800)
    if out.returncode != 0:
        raise RuntimeError(out.stderr[-2000:])
    return json.loads(out.stdout.strip().splitlines()[-1])


def cpu_sample_main(args):
    wl = WORKLOADS[args.cpu_sample]
    samples = [OracleSample(wl, 7 + b, args.cpu_heads, args.cpu_layers, args.cpu_rows, image=b,
                            nodes_sampled=args.cpu_nodes)
               for b in range(len(wl["kv_len"]))]
    times, wall = [], 0.0
    for _ in range(args.cpu_reps):
        times.append(sum(smp.run() for smp in samples))
        wall += sum(smp.wall for smp in samples)
    desc = samples[0].desc
    if len(samples) > 1:
        desc = f"per image of the {len(samples)}, summed: " + desc
    res = {"sec_per_step": times, "desc": desc, "sampled_wall_s": wall,
           "parts": {k: sum(smp.parts[k] for smp in samples) for k in samples[0].parts}}
    if args.cpu_procs > 1 and len(samples) == 1:
        # All cores: the attention sample (every head of one layer) split over
        # worker processes, one thread each, running concurrently; the step
        # time is their slowest worker x layers plus the other parts as timed
        # on one core.
        import multiprocessing as mp
        wl_h = wl["H"]
        P = min(args.cpu_procs, wl_h)
        per = [wl_h // P + (1 if i < wl_h % P else 0) for i in range(P)]
        ctx = mp.get_context("spawn")
        with ctx.Pool(P) as pool:
            pool.map(_attention_worker, [(args.cpu_sample, 7, 1, 0)] * P)  # start-up, imports
            walls = []
            for _ in range(args.cpu_reps):
                t0 = time.perf_counter()
                w = pool.map(_attention_worker, [(args.cpu_sample, 7, h, 0) for h in per], chunksize=1)
                walls.append((max(w), time.perf_counter() - t0))
        attn_layer = statistics.median(x[0] for x in walls)
        rest = samples[0].parts["expand"] + samples[0].parts["accept"] + samples[0].parts["commit"]
        res["all_core"] = {"procs": P, "attn_layer_s": attn_layer,
                           "sec_per_step": attn_layer * wl["layers"] + rest,
                           "desc": f"oracle attention of all {wl_h} heads of one layer split over {P} worker "
                                   f"processes (1 thread each, concurrent; the slowest worker's time) x "
                                   f"{wl['layers']} layers, plus expansion, rerank, walk and commit as timed "
                                   f"on one core; extrapolated to one full step"}
    print(json.dumps(res))


# ------------------------------------------------------------------ main

def decode_measure(batch, grid, fp32=False, graphs=True):
    """The end-to-end synthetic decode loop (random-init 7B-shape target and
    a one-layer EAGLE-style draft head, ADT-Tree trees every step) over a
    grid x grid image-token grid, timed as a whole, next to vanilla greedy
    decoding of the same target in plain torch (no library call; bf16
    scaled_dot_product_attention), teacher-forced with the tree decoder's
    tokens so that every emitted token is compared with the target's greedy
    choice.  Returns a dict of the measurements."""
    import torch
    from paper_2512_21857_gb300 import binding as B
    from paper_2512_21857_gb300 import build
    from paper_2512_21857_gb300.decode import Decoder, ModelShape, greedy_decode
    build.build()
    B.lib()
    shape = ModelShape(dtype=torch.float32) if fp32 else ModelShape()
    g = grid
    prompt = [int(x) for x in torch.randint(0, shape.vocab, (16,), generator=torch.Generator().manual_seed(7))]
    dec = Decoder(shape, batch=batch, grid=(g, g), prompt_len=16, seed=2025, graphs=graphs)
    # warm-up: the same grid once (cuBLAS plans, library set-up, the CUDA
    # graph of every tree size the run meets), then the timed run
    dec.generate(prompt)
    out, st = dec.generate(prompt)
    n = g * g
    van = {}
    greedy_decode(shape, dec.target_w, prompt, n, batch=batch, graphs=graphs, attn_dtype=torch.bfloat16, stats=van)
    t_van = van["seconds"]
    choice, margins = greedy_decode(shape, dec.target_w, prompt, n, batch=batch, return_margins=True, graphs=graphs,
                                    attn_dtype=torch.bfloat16, forced=out)
    diff = [(b, i) for b in range(batch) for i in range(n) if out[b][i] != choice[b][i]]
    attn = decode_verify_attention(dec, prompt_len=16, n=n)
    return {"tokens_per_s": st.tokens / st.seconds, "tau": st.tau, "accepted_draft_tokens": st.accepted,
            "accepted_length_histogram": {str(k): v for k, v in sorted(st.accept_hist.items())},
            "verify_steps": st.steps, "mean_depth": st.mean_depth, "seconds": st.seconds,
            "vanilla_greedy_tokens_per_s": batch * n / t_van,
            "speedup_vs_vanilla": (st.tokens / st.seconds) / (batch * n / t_van),
            "tokens_differing_from_target_greedy": len(diff), "tokens_checked": batch * n,
            "max_relative_top2_gap_where_differing": max((margins[b][i] for b, i in diff), default=None),
            "workload": f"random-init 7B-shape target (32 layers, hidden 4096, 32 heads x 128, SwiGLU 11008, vocab "
                        f"65536) + one-layer EAGLE-style draft head, {g}x{g} image tokens after a 16-token prompt, "
                        f"ADT-Tree controller (Anole bounds), greedy, batch {batch}",
            "dense_dtype": "fp32" if fp32 else "bf16", "launch": "CUDA graph per tree size" if graphs else "eager",
            "verify_attention": attn}


def decode_verify_attention(dec, prompt_len, n, reps=50):
    """The verify kernel at the decode loop's last cache state: the target's
    32 attention layers over each image's whole prefix (prompt + grid) for a
    64-node tree of seeded random K/V/Q, replayed back to back in a graph as
    inside the loop's step; average launch time and the share of the
    measured HBM peak its algorithmic bytes reach."""
    import torch
    from paper_2512_21857_gb300 import binding as B
    from paper_2512_21857_gb300 import synth
    tm, s = dec.target, dec.s
    Bn, N = dec.batch, 64
    L = prompt_len + n
    tb = synth.tree_batch([N] * Bn, s.vocab, 2026)
    dev = tm.device
    g = torch.Generator(device=dev)
    g.manual_seed(2026)
    layers = tm.k_cache.shape[0]
    q = (torch.randn((layers, Bn * N, s.heads, s.head_dim), generator=g, device=dev)).to(torch.bfloat16)
    kt = (torch.randn((layers, Bn * N, s.kv_heads, s.head_dim), generator=g, device=dev)).to(torch.bfloat16)
    vt = (torch.randn((layers, Bn * N, s.kv_heads, s.head_dim), generator=g, device=dev)).to(torch.bfloat16)
    out = torch.empty((Bn * N, s.heads, s.head_dim), dtype=torch.bfloat16, device=dev)
    kv_len = torch.full((Bn,), L, dtype=torch.int32, device=dev)
    parents = torch.as_tensor(tb.parents, device=dev)
    offs = torch.as_tensor(tb.node_offsets, device=dev)
    ws = B.zeroed_workspace(B.adt_tree_attn_workspace_size(Bn, s.heads, s.head_dim, N, tm.lmax), dev)
    st = torch.cuda.Stream(device=dev)

    def launch():
        for li in range(layers):
            B.adt_tree_attn(q[li], tm.k_cache[li], tm.v_cache[li], kv_len, kt[li], vt[li], parents, offs, B=Bn,
                            H=s.heads, Hkv=s.kv_heads, D=s.head_dim, max_nodes=N, max_kv=tm.lmax,
                            softmax_scale=s.head_dim ** -0.5, out=out, workspace=ws,
                            cache_stride_b=tm.k_cache.stride(1), cache_stride_h=tm.k_cache.stride(2), stream=st)

    with torch.cuda.stream(st):
        launch()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(st):
        with torch.cuda.graph(graph, stream=st):
            launch()
        for _ in range(5):
            graph.replay()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(st)
        for _ in range(reps):
            graph.replay()
        e1.record(st)
    torch.cuda.synchronize()
    us = e0.elapsed_time(e1) * 1e3 / (reps * layers)
    per_launch = Bn * (2 * L * s.kv_heads * s.head_dim * 2 + 2 * N * s.kv_heads * s.head_dim * 2
                       + 2 * N * s.heads * s.head_dim * 2)
    peak, kind = measured_peaks()
    achieved = per_launch / (us * 1e-6) / 1e9
    total = per_launch * layers
    return {"kv_len": L, "tree_nodes": N, "avg_launch_us": us, "algorithmic_bytes_per_launch": per_launch,
            "achieved_gbs": achieved, "frac": achieved / peak, "peak_source": f"{kind} (hbm_gbs)",
            "note": ("the 32 layers' prefixes total %.0f MB, less than the 129 MB L2: L2-resident, not an HBM figure"
                     % (total / 1e6)) if total < 129e6 else "inputs larger than L2"}


def run_decode(args):
    """bench.py --decode: one JSON line for the decode loop alone."""
    d = decode_measure(args.decode_batch, args.decode_grid, args.decode_fp32, not args.decode_eager)
    line = {"metric": "synthetic end-to-end decode tokens/s", "value": d.pop("tokens_per_s"), "unit": "tokens/s",
            "n_gpus": 1, "higher_is_better": True, "dtype": "bf16", "data": "synthetic (random-init weights)",
            "config": {"workload": d.pop("workload"), "batch": args.decode_batch, "dense_dtype": d.pop("dense_dtype"),
                       "launch": d.pop("launch")}}
    line.update(d)
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default="7b", choices=sorted(WORKLOADS))
    ap.add_argument("--mode", default="greedy", choices=["greedy", "spec_det"])
    ap.add_argument("--impl", default="adt", choices=["adt", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=200)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-sample", default=None)
    ap.add_argument("--cpu-heads", type=int, default=1)
    ap.add_argument("--cpu-layers", type=int, default=1)
    ap.add_argument("--cpu-rows", type=int, default=1)
    ap.add_argument("--cpu-reps", type=int, default=1)
    ap.add_argument("--cpu-nodes", type=int, default=0)
    ap.add_argument("--cpu-procs", type=int, default=1)
    ap.add_argument("--decode", action="store_true", help="the end-to-end synthetic decode loop instead")
    ap.add_argument("--decode-batch", type=int, default=1)
    ap.add_argument("--decode-grid", type=int, default=48)
    ap.add_argument("--decode-fp32", action="store_true", help="fp32 weights and residual stream in the harness")
    ap.add_argument("--decode-eager", action="store_true", help="no CUDA graphs in the decode loop")
    ap.add_argument("--no-decode", action="store_true", help="skip the decode-loop measurement of the default run")
    ap.add_argument("--bench-decode-grid", type=int, default=16,
                    help="image-token grid side of the decode-loop measurement in the default run")
    args = ap.parse_args()
    if args.decode:
        run_decode(args)
        return
    if args.cpu_sample:
        cpu_sample_main(args)
        return
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    wl = WORKLOADS[args.workload]
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    one = len(wl["kv_len"]) == 1
    config = {"workload": wl["name"], "batch": len(wl["kv_len"]), "kv_len": wl["kv_len"][0] if one else wl["kv_len"],
              "tree_nodes": wl["max_nodes"], "depth": wl["depth"][0] if one else wl["depth"],
              "width": wl["width"][0] if one else wl["width"], "vocab": wl["V"],
              "layers": wl["layers"], "heads": wl["H"], "head_dim": wl["D"], "accept_mode": args.mode,
              "l2": "inputs larger than L2: every layer reads its own 39 MB KV cache slice (1.3 GB per step)"
                    if args.workload == "7b" else
                    "inputs larger than L2: every layer reads its own KV cache slices (188 MB per layer, 6.0 GB "
                    "per step)" if args.workload == "c4" else "per-step inputs rotate through distinct layer buffers",
              "parallelism": f"replicas x{world}"}
    metric = "tree-verify steps/s"

    if args.impl == "reference":
        # The reference arm is the CPU oracle: each of the W + K steps times a
        # bounded sample of one verify step (one head of one layer of
        # attention, one draft row of expansion, the full rerank and walk,
        # one layer of KV commit) and extrapolates it to the full step.
        if rank != 0:
            return
        t_run = time.time()
        # Each step's sample shrinks with the step count so that the run stays
        # within a few minutes: past 1000 steps, attention covers a prefix of
        # the tree's nodes in proportion.
        n_steps = args.warmup + args.steps
        nodes = 0 if n_steps <= 1000 else max(4, (64 * 1000) // n_steps)
        res = cpu_sample_subprocess(args.workload, 1, 1, 1, n_steps, nodes)
        samples = res["sec_per_step"][args.warmup:]
        sec = statistics.mean(samples)
        value = 1.0 / sec
        line = {"impl": "reference", "metric": metric, "value": value, "unit": "steps/s", "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config,
                "cpu_baseline": {"kind": "oracle", "cores": 1, "sample": res["desc"], "value": value,
                                 "unit": "steps/s", "extrapolated": True,
                                 "sampled_wall_s": res["sampled_wall_s"], "cpu_model": cpu_model()},
                "extrapolated": True,
                "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
                "wall_s": time.time() - t_run}
        print(json.dumps(line), flush=True)
        return

    if world > 1:
        import torch
        torch.distributed.init_process_group("nccl")
    r = run_gpu(args, wl, rank, world)
    if rank != 0:
        if world > 1:
            import torch
            torch.distributed.destroy_process_group()
        return
    value = job_throughput(r["step_ms"], world)
    e2e_value = job_throughput(r["e2e_ms"], world)
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        if one:
            res = cpu_sample_subprocess(args.workload, wl["H"], 1, 41, 5, procs=min(os.cpu_count() or 1, 64))
        else:  # a bounded sample: 4 heads of one layer per image
            res = cpu_sample_subprocess(args.workload, 4, 1, 8, 3)
        sec = statistics.median(res["sec_per_step"])
        cpu = {"value": 1.0 / sec, "unit": "steps/s", "cores": 1, "kind": "oracle", "sample": res["desc"],
               "extrapolated": True, "sampled_wall_s": res["sampled_wall_s"], "cpu_model": cpu_model(),
               "host_cpus": os.cpu_count()}
        if "all_core" in res:
            ac = res["all_core"]
            cpu["all_core"] = {"value": 1.0 / ac["sec_per_step"], "unit": "steps/s", "cores": ac["procs"],
                               "sample": ac["desc"], "extrapolated": True}
    line = {
        "metric": metric, "value": value, "unit": "steps/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": r["step_ms"], "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": config,
        "ms_per_step_percentiles": r["step_pct"],
        "hbm_gbs_step": r["step_bytes"] / (r["step_ms"] * 1e-3) / 1e9,
        "roofline": {"bound": "hbm", "kernel": "tree_attn_tc_kernel<128>" if wl["D"] == 128 else "tree_attn_tc_kernel<64>",
                     "achieved": r["achieved"], "peak": r["peak"], "unit": "GB/s",
                     "frac": r["achieved"] / r["peak"], "peak_source": f"{r['peak_kind']} (hbm_gbs)",
                     "traffic": r["traffic"], "algorithmic_bytes_per_launch": r["attn_bytes"],
                     "avg_launch_us": r["attn_ms"] * 1e3, "kernel_sha": r["sha"]},
        "e2e": {"value": e2e_value, "unit": "steps/s", "h2d_bytes_per_step": r["h2d"],
                "d2h_bytes_per_step": r["d2h"]},
        "expansion": {"kernel": "expand_kernel", "calls_per_step": r["expand_calls"],
                      "avg_call_us": r["expand_us"],
                      "note": "image 0's draft-tree expansion calls (F = 1, then the width; the last one "
                              "without a next frontier) replayed alone back to back in a graph"},
        "gpu_launches": r["launches"],
        "clocks": r["clocks"],
        "cpu_baseline": cpu,
    }
    if world == 1 and not args.no_decode and args.workload == "7b":
        # The end-to-end decode loop (synthetic config C5) at batch 1 and 4,
        # on a bounded grid so that the default run stays within minutes.
        line["decode"] = {f"batch{bs}": decode_measure(bs, args.bench_decode_grid) for bs in (1, 4)}
    print(json.dumps(line), flush=True)
    if world > 1:
        import torch
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
