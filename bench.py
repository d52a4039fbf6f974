#!/usr/bin/env python
"""Benchmark of the Delta Attention prefill on GB300 (one JSON line, rank 0).

A step is one ``delta_attn_prefill`` call over one sequence of the seeded
synthetic workload (default: Llama-3-8B-shaped attention layer, B=1, Hq=32,
Hkv=8, d=128, N=131072, 4 sinks scaled x8, window 2048, gamma 64): the strided
dense kernel, then the sink+window kernel with the fused Delta epilogue.

  value          tokens/s of the whole job (all ranks), inputs resident in HBM
  e2e            the same through the C-ABI call on host buffers
                 (delta_attn_prefill_host): every step copies Q, K, V in and O
                 out, pipelined with the kernels per (batch, KV head) chunk
  roofline       the dominant kernel's useful TFLOP/s (unmasked pairs only, 4d
                 FLOPs per pair) against the measured bf16 peak, from CUDA events
                 recorded by the library on the launching stream
  cpu_baseline   the fp64 oracle on the host cores over a bounded sample
  dense_baseline gamma = 1 through the same kernels (dense causal attention)
  variants       the Eq. 5 "recompute" output, a dense tail block of --tail rows
                 (appendix "Implementation Details") and the three Delta
                 smoothing forms (appendix "Interpolation"), timed the same way

  workloads      (default workload only) the 32K layer and the million-token
                 prefill, each with its dense baseline, and the twelve points of
                 the B=4 window/gamma sweep, through the same timed code

The timed loop of --steps prefills is repeated back to back until the timed
region lasts about one second (each repeat bracketed by a barrier and a
device synchronize); ms_per_step is the mean over all timed steps, and the SM
clocks are sampled every 20 ms inside that region.

``--impl reference`` times the oracle as the reference arm.  Multi-GPU: one
process per GPU (torchrun), no collective on the data path; barrier + max over
ranks around each timed loop.  ``--shard replicas`` (default) runs one
independent sequence per rank (weak scaling); ``--shard heads`` splits one
prefill by (batch, KV head) pairs (strong scaling), ``--gather`` then times an
all-gather of O; ``--shard context`` splits one prefill by rows, each step
all-gathering the K and V row shards (strong scaling).
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

from paper_2505_11254_gb300 import flops  # noqa: E402
from paper_2505_11254_gb300.replicas import Replicas  # noqa: E402
from paper_2505_11254_gb300.inputs import WORKLOADS, LLAMA8B_N131K, checksums, generate, to_bits  # noqa: E402

METRIC = "Δ-attn prefill tokens/s and useful TFLOP/s (% bf16 tensor peak) at N=131K/1M"
UNIT = "tokens/s"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
KERNEL_SOURCES = ["attn_kernel.cuh", "tiles.cuh", "plan.h", "ptx.cuh", "wait.cuh", "launch_impl.cuh"]


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=40)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=LLAMA8B_N131K.name, choices=sorted(WORKLOADS))
    ap.add_argument("--window", type=int, default=None, help="override the workload's window")
    ap.add_argument("--gamma", type=int, default=None, help="override the workload's gamma")
    ap.add_argument("--cpu-seconds", type=float, default=20.0, help="oracle budget of the cpu_baseline leg")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-dense-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-variants", action="store_true", help="skip the Eq. 5 / dense-tail timings")
    ap.add_argument("--tail", type=int, default=1024, help="dense tail rows of the variant timings")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the records of the other configurations (32K, 1M, the B=4 sweep)")
    ap.add_argument("--shard", choices=["replicas", "heads", "context"], default="replicas",
                    help="N GPUs: independent sequences (weak scaling), or one prefill split by (batch, KV head) "
                         "pairs or by rows (strong scaling)")
    ap.add_argument("--gather", action="store_true", help="with --shard heads: time an all-gather of O afterwards")
    return ap.parse_args()


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f), "measured"
    return dict(PEAKS_FALLBACK), "fallback"


def _code_only(text):
    """C/C++ source without comments and blank-line or trailing-space
    differences: the part of a kernel source that decides what is compiled."""
    out, i, n = [], 0, len(text)
    while i < n:
        c = text[i]
        if c in "\"'":  # string or character literal, copied whole
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
        else:
            out.append(c)
            i += 1
    lines = (l.rstrip() for l in "".join(out).split("\n"))
    return "\n".join(l for l in lines if l)


def kernel_src_hash():
    """Hash of the attention kernels' code (comments excluded), to tell whether
    a recorded ncu traffic figure was taken on the kernels being timed."""
    h = hashlib.sha256()
    for name in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2505_11254_gb300", "csrc", name), encoding="utf-8") as f:
            h.update(_code_only(f.read()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(kernel, workload):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    the current kernel source; else None."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rec = json.load(f)
    e = rec.get(kernel, {})
    if e.get("src_sha") != kernel_src_hash() or e.get("workload") != workload:
        return None
    return e.get("dram_bytes_per_launch")


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi sampled every 20 ms while the GPU works; only the samples
    taken between mark_start() and mark_end() (host wall clock, which brackets
    the timed loops) are kept."""
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
    PERIOD_MS = 20

    def __init__(self, local_index):
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        idx = str(local_index)
        if vis:
            parts = [p.strip() for p in vis.split(",") if p.strip()]
            if local_index < len(parts):
                idx = parts[local_index]
        self.idx = idx
        self.proc = None
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits", "-i", self.idx,
                 "-lms", str(self.PERIOD_MS)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def mark_start(self):
        self.t0 = time.time()

    def mark_end(self):
        self.t1 = time.time()

    @staticmethod
    def _when(stamp):
        import datetime
        try:
            return datetime.datetime.strptime(stamp, "%Y/%m/%d %H:%M:%S.%f").timestamp()
        except ValueError:
            return None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, power, reasons, outside = [], [], [], set(), 0
        for line in out.splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 10:
                continue
            when = self._when(f[0])
            if when is not None and self.t0 is not None and not (self.t0 <= when <= (self.t1 or when)):
                outside += 1
                continue
            try:
                sm.append(float(f[2]))
                smax.append(float(f[3]))
                power.append(float(f[4]))
            except ValueError:
                continue
            for name, val in zip(self.REASONS, f[6:10]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "sm_mhz_min": min(sm) if sm else None, "power_w_max": max(power) if power else None,
                "reasons": sorted(reasons), "samples": len(sm), "period_ms": self.PERIOD_MS,
                "samples_outside_timed_region": outside}


# ------------------------------------------------------------------ oracle legs
def oracle_sample(w, Qb, Kb, Vb, budget_s, max_groups=None):
    """Time the fp64 oracle on groups of gamma rows (all query heads) at evenly
    spaced positions of the sequence.  Returns (tokens/s, seconds, groups, cores)."""
    import oracle
    n_groups_total = flops.n_samples(w.N, w.gamma)
    cores = os.cpu_count() or 1

    def run(groups):
        t0 = time.perf_counter()
        for g in groups:
            r0 = g * w.gamma
            r1 = min(r0 + w.gamma, w.N)
            oracle.delta_attn(Qb, Kb, Vb, w.n_sink, w.window, w.gamma, rows=(r0, r1), nthreads=cores)
        return time.perf_counter() - t0

    probe = [n_groups_total // 2]
    t1 = run(probe)
    m = max(1, int(budget_s / max(t1, 1e-6)))
    if max_groups:
        m = min(m, max_groups)
    m = min(m, n_groups_total)
    groups = sorted({int((i + 0.5) * n_groups_total / m) for i in range(m)})
    t = run(groups)
    rows = sum(min((g + 1) * w.gamma, w.N) - g * w.gamma for g in groups)
    return rows * w.B / t, t, len(groups), cores


def parity_spot_check(w, q, k, v, out, Qb, Kb, Vb):
    """A few output rows against the oracle (sampled and unsampled rows, early
    and late positions, the sink-dominated start)."""
    import numpy as np

    import oracle
    N, g = w.N, w.gamma
    rows = [0, 1, g, g + 5, N // 2, N // 2 + g - 1, N - g, N - 1]
    bhi = [(0, h, i) for h in (0, w.Hq - 1) for i in rows]
    ref = oracle.rows(Qb, Kb, Vb, w.n_sink, w.window, w.gamma, bhi)["A"]
    got = np.stack([out[b, h, i].double().cpu().numpy() for (b, h, i) in bhi])
    err = np.abs(got - ref)
    return {"rows": len(bhi), "max_abs": float(err.max()), "mean_abs": float(err.mean()),
            "tolerance": {"max_abs": 2e-2, "mean_abs": 2e-3}}


# ------------------------------------------------------------------ arms
def run_reference(args, w, rep):
    """Reference arm: the fp64 CPU oracle, each step a bounded sample (rank 0
    only; other ranks exit without work)."""
    if rep.rank != 0:
        return
    q, k, v = generate(w, device="cpu")
    Qb, Kb, Vb = to_bits(q), to_bits(k), to_bits(v)
    import oracle
    cores = os.cpu_count() or 1
    n_groups_total = flops.n_samples(w.N, w.gamma)
    times, rows_done = [], 0
    for s in range(args.warmup + args.steps):
        g = int((s * 0.618034 % 1.0) * n_groups_total)  # spread the sample over the sequence
        r0, r1 = g * w.gamma, min(g * w.gamma + w.gamma, w.N)
        t0 = time.perf_counter()
        oracle.delta_attn(Qb, Kb, Vb, w.n_sink, w.window, w.gamma, rows=(r0, r1), nthreads=cores)
        dt = time.perf_counter() - t0
        if s >= args.warmup:
            times.append(dt)
            rows_done += (r1 - r0) * w.B
    total = sum(times)
    value = rows_done / total
    sample = ("fp64 oracle (C, %d threads) on one group of gamma=%d rows, all %d query heads, per step, "
              "at positions spread over the %d-token sequence" % (cores, w.gamma, w.Hq, w.N))
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * total / len(times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_of(w, args.gpus),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "cpu": host_cpu(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def host_cpu():
    """Model name of the host CPU (lscpu, else /proc/cpuinfo), for the oracle's timing record."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith(("model name", "cpu part")):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return None


def config_of(w, n_gpus, shard="replicas"):
    qkv = 2 * w.d * w.N * (w.B * w.Hq + 2 * w.B * w.Hkv)
    l2 = ("inputs larger than L2 (Q+K+V %.2f GiB vs 129 MB L2), no flush" % (qkv / 2 ** 30) if qkv > 129e6 else
          "inputs smaller than L2 (%.1f MB), no flush: not a headline configuration" % (qkv / 1e6))
    return {"workload": w.name, "B": w.B, "Hq": w.Hq, "Hkv": w.Hkv, "d": w.d, "N": w.N, "n_sink": w.n_sink,
            "window": w.window, "gamma": w.gamma, "rope_base": w.rope_base if w.rope else None,
            "sink_scale": w.sink_scale,
            "l2": l2,
            "parallelism": ("single GPU" if n_gpus == 1 else
                            "head shards: one prefill, (batch, KV head) pairs split over %d GPUs" % n_gpus
                            if shard == "heads" else "replicas: one independent sequence per GPU")}


def time_variants(args, w, q, k, v, out, stream, restore):
    """Median CUDA-event time of the prefill in the paper's ablation forms:
    recompute (Eq. 5), Delta with a dense tail, recompute with a dense tail,
    and the smoothed corrections (linear, EMA beta 0.5, the filter with
    (0.2, 0.05, 0.0035)).  The inputs are larger than L2, as in the main loop."""
    from paper_2505_11254_gb300 import binding
    res = {}
    for name, mode, tail, sm, par in (("recompute", "recompute", 0, "none", ()),
                                      ("delta_tail", "delta", args.tail, "none", ()),
                                      ("recompute_tail", "recompute", args.tail, "none", ()),
                                      ("smooth_linear", "delta", 0, "linear", ()),
                                      ("smooth_ema", "delta", 0, "ema", (0.5,)),
                                      ("smooth_abg", "delta", 0, "abg", (0.2, 0.05, 0.0035))):
        ws = binding.alloc_workspace(binding.workspace_size(w.B, w.Hq, w.Hkv, w.N, w.d, w.n_sink, w.window,
                                                            w.gamma, mode, tail, smooth=sm), q.device)

        def call():
            binding.delta_attn_prefill(q, k, v, w.n_sink, w.window, w.gamma, out=out, workspace=ws, mode=mode,
                                       tail_dense=tail, smooth=sm, smooth_params=par)
        for _ in range(3):
            call()
        torch.cuda.synchronize()
        times = []
        for _ in range(10):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            call()
            e1.record(stream)
            torch.cuda.synchronize()
            times.append(e0.elapsed_time(e1))
        if binding.check() != binding.DA_OK:
            raise RuntimeError("device status after the %s timing" % name)
        ms = statistics.median(times)
        res[name] = {"mode": mode, "tail_dense": tail, "smooth": sm, "smooth_params": list(par), "ms": ms,
                     "tokens_per_s": w.B * w.N / (ms / 1e3),
                     "tail_dense_pairs_per_head": flops.tail_pairs_per_head(w.N, tail)}
        del ws
    res["rope_prefill"] = time_rope_prefill(w, q, k, v, out, stream)
    res["standalone"] = time_standalone(w, q, k, v, stream)
    res["decode"] = time_decode(w, q, k, v, stream)
    restore()  # `out` back to the Delta result for the spot check
    return res


def time_rope_prefill(w, q, k, v, out, stream):
    """The prefill with RoPE fused (delta_attn_prefill_rope): K rotated in
    place by a pass of its own, each Q tile rotated on its way into tensor
    memory.  Timed on a copy of K, restored before every call, outside the
    timed region."""
    from paper_2505_11254_gb300 import binding
    table = binding.rope_table(w.N, w.d, 500000.0, device=q.device)
    kc = torch.empty_like(k)
    ws = binding.alloc_workspace(binding.workspace_size(w.B, w.Hq, w.Hkv, w.N, w.d, w.n_sink, w.window, w.gamma),
                                 q.device)
    times = []
    for it in range(13):
        kc.copy_(k)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        binding.delta_attn_prefill_rope(q, kc, v, w.n_sink, w.window, w.gamma, table, out=out, workspace=ws)
        e1.record(stream)
        torch.cuda.synchronize()
        if it >= 3:
            times.append(e0.elapsed_time(e1))
    if binding.check() != binding.DA_OK:
        raise RuntimeError("device status after the RoPE prefill timing")
    ms = statistics.median(times)
    return {"ms": ms, "tokens_per_s": w.B * w.N / (ms / 1e3), "rope_base": 500000.0,
            "note": "K rotated in place (one pass), Q rotated inside the attention kernels"}


def time_standalone(w, q, k, v, stream):
    """The three parts through their own entry points, the unfused order of
    Alg. 1: sparse_window_attn (bf16 S and the fp32 sparse rows at the
    samples), strided_dense_attn (fp32 dense rows at the samples), then
    delta_apply adding Delta_k to every row in place (one more read and write
    of O than the fused prefill).  Median over 10 calls after 3 warm-ups, with
    events between the three calls; delta_apply's bytes (O read and written
    in bf16, both sampled-row sets read in fp32) against the measured HBM copy
    bandwidth."""
    from paper_2505_11254_gb300 import binding
    peaks, _ = load_peaks()
    ns = -(-w.N // w.gamma)
    o = torch.empty_like(q)
    s_s = torch.empty((w.B, w.Hq, ns, w.d), dtype=torch.float32, device=q.device)
    d_s = torch.empty_like(s_s)
    dws = binding.alloc_workspace(binding.strided_dense_workspace_size(w.B, w.Hq, w.Hkv, w.N, w.d, w.gamma),
                                  q.device)

    def call(evs):
        evs[0].record(stream)
        binding.sparse_window_attn(q, k, v, w.n_sink, w.window, w.gamma, out=o, s_sampled=s_s)
        evs[1].record(stream)
        binding.strided_dense_attn(q, k, v, w.gamma, out=d_s, workspace=dws)
        evs[2].record(stream)
        binding.delta_apply(o, s_s, d_s, w.gamma, out=o)
        evs[3].record(stream)

    rows = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(13)]
    for r in rows:
        call(r)
    torch.cuda.synchronize()
    if binding.check() != binding.DA_OK:
        raise RuntimeError("device status after the standalone timing")
    rows = rows[3:]
    parts = {name: statistics.median(r[i].elapsed_time(r[i + 1]) for r in rows)
             for i, name in enumerate(("sparse_window_attn", "strided_dense_attn", "delta_apply"))}
    total = statistics.median(r[0].elapsed_time(r[3]) for r in rows)
    apply_bytes = 2 * w.B * w.Hq * w.N * w.d * 2 + 2 * w.B * w.Hq * ns * w.d * 4
    hbm = float(peaks.get("hbm_gbs", PEAKS_FALLBACK["hbm_gbs"]))
    gbs = apply_bytes / (parts["delta_apply"] / 1e3) / 1e9
    return {"ms": total, "tokens_per_s": w.B * w.N / (total / 1e3), "parts_ms": parts,
            "delta_apply_bytes": apply_bytes, "delta_apply_gbs": gbs, "delta_apply_frac_of_hbm": gbs / hbm,
            "note": "three entry points; the fused prefill writes O once instead"}


def time_decode(w, q, k, v, stream):
    """Eq. 2 decoding of one new token per sequence over the whole N-token
    cache (the workload's K and V; the last row plays the new token's key and
    value).  ``ms`` is the device time per call of 20 back-to-back calls that
    alternate between two copies of the cache, so that no call finds the
    previous call's keys in L2 (each copy is several times the L2); the K/V
    bytes a call must read (each cached byte once) are set against the
    measured HBM copy bandwidth.  ``ms_synchronous`` is one call bracketed by
    events with a synchronize after it: host-side launch latency included."""
    from paper_2505_11254_gb300 import binding
    peaks, _ = load_peaks()
    qd = q[:, :, -1, :].contiguous()
    caches = [(k, v), (k.clone(), v.clone())]
    ws = binding.alloc_workspace(binding.decode_workspace_size(w.B, w.Hq, w.Hkv, w.N, w.d), q.device)
    od = torch.empty_like(qd)
    for i in range(4):
        binding.decode(qd, *caches[i % 2], out=od, workspace=ws)
    torch.cuda.synchronize()
    reps, blocks = 20, []
    for _ in range(5):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(reps):
            binding.decode(qd, *caches[i % 2], out=od, workspace=ws)
        e1.record(stream)
        torch.cuda.synchronize()
        blocks.append(e0.elapsed_time(e1) / reps)
    single = []
    for i in range(10):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        binding.decode(qd, *caches[i % 2], out=od, workspace=ws)
        e1.record(stream)
        torch.cuda.synchronize()
        single.append(e0.elapsed_time(e1))
    if binding.check() != binding.DA_OK:
        raise RuntimeError("device status after the decode timing")
    del caches
    ms = statistics.median(blocks)
    kv_bytes = 2 * w.B * w.Hkv * w.N * w.d * 2
    gbs = kv_bytes / (ms / 1e3) / 1e9
    hbm = float(peaks.get("hbm_gbs", PEAKS_FALLBACK["hbm_gbs"]))
    return {"context": w.N, "ms": ms, "ms_synchronous": statistics.median(single),
            "tokens_per_s": w.B / (ms / 1e3), "kv_bytes": kv_bytes,
            "achieved_gbs": gbs, "hbm_peak_gbs": hbm, "frac_of_hbm": gbs / hbm,
            "note": "one token per sequence, all heads; split-K kernel + merge kernel (dependent launch) per call"}


KERNEL_NAMES = {1: ["dense_bf16"], 2: ["strided_dense_f32", "sink_window_fused_delta"],
                3: ["strided_dense_f32", "strided_sparse_delta", "sink_window_delta"]}


def kernel_flops(w, nk):
    """Useful FLOPs of each kernel of the launch sequence (4d per unmasked
    pair: the dense rows in the strided dense kernel, the sink+window rows in
    the sink+window kernel; the strided sparse Delta pass adds none)."""
    hq_flops = 4 * w.d * w.B * w.Hq
    dense_f = hq_flops * flops.dense_pairs_per_head(w.N, w.gamma)
    sparse_f = hq_flops * flops.sparse_pairs_per_head(w.N, w.n_sink, w.window)
    return {1: [dense_f], 2: [dense_f, sparse_f], 3: [dense_f, 0, sparse_f]}[nk]


def time_prefill(w, q, k, v, steps, warmup, rep, peaks, peak_src, local, min_seconds=1.0, max_repeats=25):
    """Warm-up, then the timed loop of `steps` delta_attn_prefill calls,
    repeated back to back (each repeat bracketed by a barrier and a device
    synchronize, the max over ranks taken per repeat) until the timed region
    lasts about `min_seconds` (about 50 clock samples at one per 20 ms).
    A second loop of as many calls, right after, has the library record CUDA
    events between its kernels on the launching stream: those give the
    per-kernel times (each kernel then runs alone, without the overlap of a
    programmatic dependent launch).  Returns (record, out) with out holding
    the last step's result."""
    from paper_2505_11254_gb300 import binding
    B, Hq, Hkv, N, d = q.shape[0], q.shape[1], k.shape[1], q.shape[2], q.shape[3]
    info = binding.plan_info(B, Hq, Hkv, N, d, w.n_sink, w.window, w.gamma)
    nk = int(info["kernels"])
    ws = binding.alloc_workspace(binding.workspace_size(B, Hq, Hkv, N, d, w.n_sink, w.window, w.gamma), q.device)
    out = torch.empty_like(q)
    stream = torch.cuda.current_stream()

    def step(evs=None):
        if evs is None:
            binding.delta_attn_prefill(q, k, v, w.n_sink, w.window, w.gamma, out=out, workspace=ws)
        else:
            binding.delta_attn_prefill_events(q, k, v, w.n_sink, w.window, w.gamma, evs, out=out, workspace=ws)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    status = binding.check()
    if status != binding.DA_OK:
        raise RuntimeError("device status %d after warm-up" % status)
    # length of one step, to size the number of repeats of the timed loop
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    step()
    e1.record(stream)
    torch.cuda.synchronize()
    est_ms = rep.max(e0.elapsed_time(e1))
    repeats = max(1, min(max_repeats, int(-(-min_seconds * 1e3 // (steps * est_ms)))))

    n_ev = min(steps * repeats, max(steps, 40))
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(nk + 1)] for _ in range(n_ev)]
    for row in evs:
        for e in row:
            e.record(stream)  # create the events before the timed region
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    for _ in range(3):  # keep the GPU busy while the sampler starts
        step()
    time.sleep(0.25)
    loop_ms = []
    clocks.mark_start()
    for r in range(repeats):
        rep.barrier()
        torch.cuda.synchronize()
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for s in range(steps):
            step()
        t_end.record(stream)
        torch.cuda.synchronize()
        rep.barrier()
        loop_ms.append(rep.max(t_start.elapsed_time(t_end)))
    clocks.mark_end()
    for row in evs:  # per-kernel times
        step(row)
    torch.cuda.synchronize()
    clock_info = clocks.stop()
    status = binding.check()
    if status != binding.DA_OK:
        raise RuntimeError("device status %d after the timed loop" % status)

    ms_per_step = sum(loop_ms) / (repeats * steps)
    names = KERNEL_NAMES[nk]
    kt = [statistics.mean(row[i].elapsed_time(row[i + 1]) for row in evs) for i in range(nk)]
    kflops = kernel_flops(w.with_(B=B, Hq=Hq, N=N, d=d), nk)
    kernels = [{"name": n, "ms": t, "share": t / sum(kt), "useful_tflops": (f / (t / 1e3) / 1e12) if f else None}
               for n, t, f in zip(names, kt, kflops)]
    dom = max(range(nk), key=lambda i: kt[i])
    peak = float(peaks.get("bf16_tflops", PEAKS_FALLBACK["bf16_tflops"]))
    achieved = kflops[dom] / (kt[dom] / 1e3) / 1e12 if kflops[dom] else None
    roofline = {"bound": "tensor", "kernel": names[dom], "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": (achieved / peak) if achieved else None, "traffic": recorded_traffic(names[dom], w.name),
                "peak_source": "%s bf16 dense burst (MEASURED_PEAKS.json)" % peak_src if peak_src == "measured"
                else "fallback 1.9 PFLOP/s bf16",
                "algorithmic": "4*d FLOPs per unmasked (query, key) pair: %.4g FLOP per launch" % kflops[dom]}
    total_f = flops.useful_flops(B, Hq, N, d, w.n_sink, w.window, w.gamma)
    useful_tflops = total_f / (ms_per_step / 1e3) / 1e12
    sustained = float(peaks.get("bf16_tflops_sustained", PEAKS_FALLBACK["bf16_tflops_sustained"]))
    rec = {"ms_per_step": ms_per_step, "median_ms_per_step": statistics.median(loop_ms) / steps,
           "timed_repeats": repeats, "loop_ms": loop_ms,
           "useful_tflops": useful_tflops, "pct_of_bf16_peak": 100 * useful_tflops / peak,
           "pct_of_bf16_sustained": 100 * useful_tflops / sustained, "roofline": roofline, "kernels": kernels,
           "gpu_launches": nk * steps * repeats, "clocks": clock_info}
    return rec, out, step


def time_dense_baseline(w, q, k, v, reps, ms_delta):
    """gamma = 1 through the same kernels: every row a dense causal row (the
    quadratic baseline of the paper's latency figures)."""
    from paper_2505_11254_gb300 import binding
    stream = torch.cuda.current_stream()
    dws = binding.alloc_workspace(binding.workspace_size(w.B, w.Hq, w.Hkv, w.N, w.d, w.n_sink, w.window, 1),
                                  q.device)
    out = torch.empty_like(q)
    d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    d0.record(stream)
    for _ in range(reps):
        binding.delta_attn_prefill(q, k, v, w.n_sink, w.window, 1, out=out, workspace=dws)
    d1.record(stream)
    torch.cuda.synchronize()
    if binding.check() != binding.DA_OK:
        raise RuntimeError("device status after the dense baseline")
    dense_ms = d0.elapsed_time(d1) / reps
    dflops = flops.dense_flops(w.B, w.Hq, w.N, w.d)
    return {"ms": dense_ms, "reps": reps, "tflops": dflops / (dense_ms / 1e3) / 1e12,
            "speedup_of_delta": dense_ms / ms_delta,
            "note": "gamma=1 through the same kernels = dense causal attention"}


def time_workloads(args, dev, rep, peaks, peak_src):
    """The other configurations, through the same timed code as the headline
    (rank 0, one GPU): the 32K layer, the million-token prefill with its
    dense causal baseline, and the twelve points of the B=4 window/gamma sweep
    (one set of inputs; window and gamma change only the kernels' work)."""
    from paper_2505_11254_gb300.inputs import LLAMA8B_N1M, LLAMA8B_N32K, SWEEP_B4_N64K, SWEEP_GAMMAS, SWEEP_WINDOWS
    res = {}

    def one(w, q, k, v, dense_reps=0):
        rec, out, _ = time_prefill(w, q, k, v, min(args.steps, 10), 3, rep, peaks, peak_src, rep.local)
        rec.update({"tokens_per_s": w.B * w.N / (rec["ms_per_step"] / 1e3), "config": config_of(w, 1),
                    "input_checksums": checksums(q, k, v)})
        for key in ("loop_ms",):
            rec.pop(key, None)
        del out
        if dense_reps:
            rec["dense_baseline"] = time_dense_baseline(w, q, k, v, dense_reps, rec["ms_per_step"])
        return rec

    for w, dense_reps in ((LLAMA8B_N32K, 0 if args.no_dense_baseline else 3),
                          (LLAMA8B_N1M, 0 if args.no_dense_baseline else 1)):
        q, k, v = generate(w, device=dev)
        res[w.name] = one(w, q, k, v, dense_reps)
        del q, k, v
        torch.cuda.empty_cache()
    q, k, v = generate(SWEEP_B4_N64K, device=dev)
    sweep = {}
    for window in SWEEP_WINDOWS:
        for gamma in SWEEP_GAMMAS:
            sweep["w%d_g%d" % (window, gamma)] = one(SWEEP_B4_N64K.with_(window=window, gamma=gamma), q, k, v)
    res[SWEEP_B4_N64K.name] = sweep
    del q, k, v
    torch.cuda.empty_cache()
    return res


def run_context(args, w, rep):
    """One prefill split by rows over the ranks (context parallelism): a step
    is the all-gather of the K and V row shards and delta_attn_prefill_rows on
    this rank's rows; barrier and max over ranks around the timed loop."""
    from paper_2505_11254_gb300 import binding
    from paper_2505_11254_gb300.replicas import context_shard, gather_kv
    world, rank, local = rep.world, rep.rank, rep.local
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    q_all, k_all, v_all = generate(w, device=dev)
    r0, r1 = context_shard(w.N, w.gamma, rank, world)
    if r1 <= r0:
        raise RuntimeError("rank %d has no rows: use at most %d GPUs" % (rank, -(-w.N // 128)))
    q = q_all[:, :, r0:r1].contiguous()
    k_own, v_own = k_all[:, :, r0:r1].contiguous(), v_all[:, :, r0:r1].contiguous()
    del q_all, k_all, v_all
    ws = binding.alloc_workspace(binding.workspace_size_rows(w.B, w.Hq, w.Hkv, w.N, w.d, w.n_sink, w.window,
                                                             w.gamma, r0, r1 - r0), dev)
    out = torch.empty_like(q)
    nk = int(binding.plan_info(w.B, w.Hq, w.Hkv, w.N, w.d, w.n_sink, w.window, w.gamma)["kernels"])

    def step():
        k, v = gather_kv(k_own, v_own, w.N, w.gamma, world) if world > 1 else (k_own, v_own)
        binding.delta_attn_prefill_rows(q, k, v, w.n_sink, w.window, w.gamma, r0, out=out, workspace=ws)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if binding.check() != binding.DA_OK:
        raise RuntimeError("device status after warm-up")
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.25)
    clocks.mark_start()
    rep.barrier()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(args.steps):
        step()
    t1.record()
    torch.cuda.synchronize()
    rep.barrier()
    clocks.mark_end()
    clock_info = clocks.stop()
    if binding.check() != binding.DA_OK:
        raise RuntimeError("device status after the timed loop")
    ms_per_step = rep.max(t0.elapsed_time(t1)) / args.steps
    peaks, _ = load_peaks()
    peak = float(peaks.get("bf16_tflops", PEAKS_FALLBACK["bf16_tflops"]))
    useful = flops.useful_flops(w.B, w.Hq, w.N, w.d, w.n_sink, w.window, w.gamma) / (ms_per_step / 1e3) / 1e12
    if rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": w.B * w.N / (ms_per_step / 1e3), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "strong", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic: seeded N(0,1) Q,K,V, RoPE base 500000 on Q,K, sink keys x%g; no dataset"
                    % w.sink_scale,
            "config": dict(config_of(w, world), parallelism="context shards: one prefill split by rows over %d GPUs"
                           " (all-gather of the K, V row shards each step)" % world),
            "useful_tflops": useful, "pct_of_bf16_peak": 100 * useful / peak, "rows": [r0, r1],
            "gpu_launches": nk * args.steps, "clocks": clock_info}), flush=True)


def run_ours(args, w, rep):
    from paper_2505_11254_gb300 import binding
    from paper_2505_11254_gb300.replicas import head_shard, shard_views, gather_shards
    world, rank, local = rep.world, rep.rank, rep.local
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    peaks, peak_src = load_peaks()
    sharded = args.shard == "heads"
    if sharded:
        # one prefill, its (batch, KV head) pairs split over the ranks
        q_all, k_all, v_all = generate(w, device=dev)
        p0, p1 = head_shard(w.B, w.Hkv, rank, world)
        if p1 <= p0:
            raise RuntimeError("rank %d has no (batch, KV head) pair: use at most %d GPUs" % (rank, w.B * w.Hkv))
        q, k, v = (t.contiguous() for t in shard_views(q_all, k_all, v_all, w.Hkv, p0, p1))
        ws_ = w.with_(name=w.name + "_shard", B=p1 - p0, Hq=w.Hq // w.Hkv, Hkv=1)
    else:
        wr = w.with_(seed=rep.seed(w.seed))
        q, k, v = generate(wr, device=dev)
        ws_ = w
    rec, out, step = time_prefill(ws_, q, k, v, args.steps, args.warmup, rep, peaks, peak_src, local)
    ms_per_step = rec["ms_per_step"]
    tokens_per_step = w.B * w.N
    value = (tokens_per_step / (ms_per_step / 1e3)) if sharded else rep.throughput(tokens_per_step,
                                                                                   ms_per_step / 1e3)
    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "strong" if sharded else "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: seeded N(0,1) Q,K,V, RoPE base 500000 on Q,K, sink keys x%g; no dataset" % w.sink_scale,
        "config": config_of(w, world, args.shard),
    }
    result.update({key: rec[key] for key in ("useful_tflops", "pct_of_bf16_peak", "pct_of_bf16_sustained",
                                             "roofline", "kernels", "gpu_launches", "clocks", "timed_repeats",
                                             "loop_ms", "median_ms_per_step")})
    result["input_checksums"] = checksums(q, k, v)
    if sharded:
        result["useful_tflops"] = flops.useful_flops(w.B, w.Hq, w.N, w.d, w.n_sink, w.window, w.gamma) / (
            ms_per_step / 1e3) / 1e12
        result["shard"] = {"pairs": [p0, p1], "of_pairs": w.B * w.Hkv}
        if world > 1 and args.gather:
            torch.cuda.synchronize()
            rep.barrier()
            g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            g0.record()
            gather_shards(out, w.B, w.Hq, w.Hkv, world)
            g1.record()
            torch.cuda.synchronize()
            result["shard"]["gather_ms"] = rep.max(g0.elapsed_time(g1))

    if not args.no_e2e and not sharded:
        # End to end through the C-ABI call on HOST buffers (page-locked):
        # every step copies Q, K, V in and O out; the call pipelines the
        # copies with the kernels per (batch, KV head) chunk.
        stream = torch.cuda.current_stream()
        qh, kh, vh = (t.cpu().pin_memory() for t in (q, k, v))
        oh = torch.empty(out.shape, dtype=out.dtype, pin_memory=True)
        hws = binding.alloc_workspace(binding.host_workspace_size(w.B, w.Hq, w.Hkv, w.N, w.d, w.n_sink, w.window,
                                                                  w.gamma), dev)

        def e2e_step():
            binding.delta_attn_prefill_host(qh, kh, vh, w.n_sink, w.window, w.gamma, out=oh, workspace=hws)

        for _ in range(max(1, args.warmup)):
            e2e_step()
        torch.cuda.synchronize()
        rep.barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            e2e_step()
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = rep.max(e0.elapsed_time(e1)) / args.steps
        if binding.check() != binding.DA_OK:
            raise RuntimeError("device status after the e2e loop")
        result["e2e"] = {"value": rep.throughput(tokens_per_step, e2e_ms / 1e3), "unit": UNIT,
                         "h2d_bytes_per_step": sum(t.numel() * t.element_size() for t in (q, k, v)),
                         "d2h_bytes_per_step": out.numel() * out.element_size(), "ms_per_step": e2e_ms}
        result["e2e"]["path"] = "delta_attn_prefill_host (host buffers, copies pipelined per KV-head chunk)"
        del qh, kh, vh, oh, hws

    solo = rank == 0 and not sharded
    if not args.no_dense_baseline and solo:
        result["dense_baseline"] = time_dense_baseline(w, q, k, v, 3, ms_per_step)

    if not args.no_variants and solo:
        result["variants"] = time_variants(args, w, q, k, v, out, torch.cuda.current_stream(), step)

    if solo and world == 1 and not args.no_cpu_baseline:
        torch.cuda.synchronize()
        Qb, Kb, Vb = to_bits(q), to_bits(k), to_bits(v)
        result["parity"] = parity_spot_check(w, q, k, v, out, Qb, Kb, Vb)
        tps, secs, groups, cores = oracle_sample(w, Qb, Kb, Vb, args.cpu_seconds)
        result["cpu_baseline"] = {
            "value": tps, "unit": UNIT, "cores": cores, "cpu": host_cpu(), "kind": "oracle",
            "sample": "%d groups of gamma=%d rows x all %d query heads at evenly spaced positions of the "
                      "%d-token sequence, fp64 C oracle on %d threads, %.1f s" % (
                          groups, w.gamma, w.Hq, w.N, cores, secs)}
        del Qb, Kb, Vb

    if solo and world == 1 and not args.no_workloads and w.name == LLAMA8B_N131K.name:
        del q, k, v, out
        torch.cuda.empty_cache()
        result["workloads"] = time_workloads(args, dev, rep, peaks, peak_src)
    if rank == 0:
        print(json.dumps(result), flush=True)


def main():
    args = parse_args()
    w = WORKLOADS[args.workload]
    if args.window is not None:
        w = w.with_(window=args.window)
    if args.gamma is not None:
        w = w.with_(gamma=args.gamma)
    rep = Replicas().init()
    try:
        if args.impl == "reference":
            run_reference(args, w, rep)
        elif args.shard == "context":
            run_context(args, w, rep)
        else:
            run_ours(args, w, rep)
    finally:
        rep.close()


if __name__ == "__main__":
    main()
