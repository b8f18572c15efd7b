"""Decode-step benchmark of the MLKV decode-attention library.

One step = for every layer n in order: store the new token (owner layers only) then attend --
mlkv_append_decode_attention(n) for owner layers (one launch for both), mlkv_decode_attention(n)
for the others.  Default workload: Pythia-160M-shaped
MLKV-2 (12 layers, 12 query heads, head_dim 64, owner layers 0 and 6 with one KV head each),
batch 64, context 2048, bf16 Q/K/V ~ N(0,1) from a seeded generator.

value   decode tokens/s of the whole job = batch * world / step time; device time of one
        mlkv_decode_step call (the library replays the step's launches from a CUDA graph), CUDA
        events on the launching stream, L2 flushed (a 512 MiB write) before every step outside
        the timed events.
e2e     the same metric end to end through the C ABI with host buffers: one
        mlkv_decode_step_host call per step (the step's Q and new K/V copied from pinned host
        memory, every layer's decode, every layer's output copied back), inside the timed region;
        queued behind the L2 flush like the device-timed steps, the host waiting for each step's
        outputs before the next.
roofline  the decode kernel: logical K/V bytes per launch / mean launch duration (CUDA events
        around each launch) against the measured HBM copy bandwidth.
cpu_baseline  the fp64 oracle (test infrastructure) on the host cores, on a bounded sample.

--impl reference times the oracle alone (the reference arm for this workload).
Multi-GPU (torchrun): every rank runs an independent replica; no collective touches the data.
"""
import argparse
import json
import math
import os
import statistics
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "decode-attn tokens/s per step (all layers); HBM GB/s vs GB300 peak"
UNIT = "tokens/s"
DEFAULT_WORKLOAD = "pythia160m-mlkv2-b64-L2048"
FLUSH_BYTES = 512 << 20


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def max_over_ranks(ms, dist, device):
    """The job's step time: the slowest rank's (every rank runs a whole replica, weak scaling)."""
    if dist is None:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(batch, world, ms):
    """Whole-job tokens per second: every rank's batch over the slowest rank's step time."""
    return batch * world / (ms / 1e3)


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


class Clocks:
    """Samples the SM clock and the clock-event (throttle) reasons through NVML while the timed
    region runs: a background thread polls every few milliseconds, plus one sample at entry and
    one at exit.  Read-only queries; no setting of the GPU is changed."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, index, period_s=0.005):
        import ctypes
        import threading
        self.period = period_s
        self.samples = []
        self.max_mhz = None
        self.stop = threading.Event()
        self.thread = None
        self.nvml = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            if nv.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(index), ctypes.byref(h)) != 0:
                return
            self.nvml, self.h = nv, h
            mx = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = float(mx.value)
            fn = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None)
            self.reason_fn = fn or nv.nvmlDeviceGetCurrentClocksThrottleReasons
        except Exception:
            self.nvml = None

    def _sample(self):
        import ctypes
        c = ctypes.c_uint()
        r = ctypes.c_ulonglong()
        if self.nvml.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(c)) != 0:
            return
        self.reason_fn(self.h, ctypes.byref(r))
        self.samples.append((float(c.value), int(r.value)))

    def _loop(self):
        while not self.stop.wait(self.period):
            self._sample()

    def __enter__(self):
        import threading
        if self.nvml is not None:
            self._sample()
            self.thread = threading.Thread(target=self._loop, daemon=True)
            self.thread.start()
        return self

    def __exit__(self, *exc):
        if self.nvml is not None:
            self.stop.set()
            self.thread.join()
            self._sample()
        return False

    def summary(self):
        if not self.samples:
            return None
        reasons = set()
        for _, r in self.samples:
            for bit, name in self.REASONS.items():
                if r & bit:
                    reasons.add(name)
        return {"sm_mhz": statistics.median(c for c, _ in self.samples),
                "sm_max_mhz": self.max_mhz, "reasons": sorted(reasons),
                "samples": len(self.samples), "source": "nvml"}


def oracle_sample(w, rows, nthreads, reps=1):
    """Runs the oracle over every layer of the workload for the first `rows` sequences, `reps`
    decode steps in a row.

    Returns (wall seconds, CPU seconds of all threads, sequences processed).  Inputs are the
    generator's values, built before the clock starts."""
    import oracle
    from mlkv_synth import gen

    seq_lens = w.seq_lens()[:rows]
    L = int(seq_lens.max())
    betas = list(range(rows))
    caches = {}
    for n in w.owners():
        k = gen.bf16_bits_to_f64(gen.gen_kv(w.seed, n, 0, w.b, w.g, L, w.d, w.sigma_k, betas))
        v = gen.bf16_bits_to_f64(gen.gen_kv(w.seed, n, 1, w.b, w.g, L, w.d, w.sigma_v, betas))
        caches[n] = (k, v)
    qs = [gen.bf16_bits_to_f64(gen.gen_q(w.seed, n, w.b, w.h, w.d, w.sigma_q, betas))
          for n in range(w.l)]
    c0, t0 = time.process_time(), time.perf_counter()
    for _ in range(reps):
        for n in range(w.l):
            k, v = caches[w.owner[n]]
            oracle.decode_layer(n, w.owner, w.h, w.g, w.d, seq_lens, qs[n], k, v, nthreads)
    return time.perf_counter() - t0, time.process_time() - c0, rows * reps


def cpu_baseline(w, budget_cpu_s=15.0):
    """Times the oracle as it stands on this host's cores over a bounded sample: the first
    sequences of the batch, grown toward about `budget_cpu_s` of CPU time, then whole decode
    steps repeated while the full batch stays below it."""
    nthreads = os.cpu_count() or 1
    rows = max(1, min(w.b, nthreads))
    t, c, r = oracle_sample(w, rows, nthreads)
    # grow the sample toward the budget (the oracle's cost is linear in sequences)
    if c < budget_cpu_s / 4 and rows < w.b:
        rows = int(min(w.b, max(rows + 1, rows * budget_cpu_s / 2 / max(c, 1e-3))))
        t, c, r = oracle_sample(w, rows, nthreads)
    reps = 1
    if c < budget_cpu_s / 4 and rows == w.b:
        reps = int(min(1000, math.ceil(budget_cpu_s / max(c, 1e-3))))
        t, c, r = oracle_sample(w, rows, nthreads, reps)
    steps = f"{reps} decode steps" if reps > 1 else "one decode step"
    return {"value": r / t, "unit": UNIT, "cores": nthreads, "kind": "oracle",
            "sample": f"first {rows} of {w.b} sequences, all {w.l} layers, {steps} "
                      f"({t:.2f} s wall, {c:.1f} s CPU); tokens/s = sequences / oracle seconds"}


def run_reference(args, w):
    world, rank, _ = _dist()
    if rank != 0:
        return
    nthreads = os.cpu_count() or 1
    rows = max(1, min(w.b, nthreads))
    for _ in range(args.warmup):
        oracle_sample(w, rows, nthreads)
    times = []
    for _ in range(args.steps):
        t, _, _ = oracle_sample(w, rows, nthreads)
        times.append(t)
    t = sum(times) / len(times)
    value = rows / t
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "impl": "reference", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": _config_dict(w),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": nthreads, "kind": "oracle",
                         "sample": f"first {rows} of {w.b} sequences, all {w.l} layers per step"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def _config_dict(w):
    return {"workload": w.name, "layers": w.l, "q_heads": w.h, "head_dim": w.d,
            "layer_owner": w.owner, "kv_heads_per_owner": w.g, "batch": w.b,
            "context": "uniform[1,%d]" % w.L if w.uniform_len else w.L,
            "l2": "flushed before every timed step (512 MiB write)", "parallelism": "replicas"}


# What each kernel is built from (the fused decode is the prefill kernel's fused form).
KERNEL_SOURCES = {
    "decode_kernel": ("mlkv_kernels.cu", "mlkv_device.cuh"),
    "prefill_kernel": ("mlkv_prefill.cu", "mlkv_tcgen05.cuh", "mlkv_device.cuh"),
}


def _kernel_source_hash(kernel="decode_kernel"):
    """sha256[:16] over a kernel's sources, in KERNEL_SOURCES order, with comments, trailing
    blanks and empty lines removed (so that a capture stays valid while only comments change)."""
    import hashlib
    import re
    h = hashlib.sha256()
    for name in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2406_09297_gb300", "csrc", name)) as f:
            text = f.read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        lines = [ln.rstrip() for ln in text.splitlines()]
        h.update("\n".join(ln for ln in lines if ln).encode())
    return h.hexdigest()[:16]


def _recorded_traffic(w, kernel, launch):
    """DRAM bytes per launch of the step's dominant kernel (dram__bytes_read.sum +
    dram__bytes_write.sum) from the ncu capture recorded in profiles/decode_traffic.json for this
    workload, kernel and step form ("multi-layer": one decode launch for the step, "fused": the
    cross-layer fused form, "per-layer"), or None when there is none or the kernel's sources
    changed since it was taken."""
    try:
        with open(os.path.join(ROOT, "profiles", "decode_traffic.json")) as f:
            rec = json.load(f)
    except Exception:
        return None
    if kernel not in KERNEL_SOURCES:
        return None
    for entry in rec.get("entries", []):
        if (entry.get("workload") == w.name and entry.get("kernel") == kernel and
                entry.get("launch") == launch and
                entry.get("kernel_source_sha256_16") == _kernel_source_hash(kernel)):
            return entry.get("dram_bytes_per_launch")
    return None


def kv_bytes_per_layer(w, seq_lens):
    return int(np.sum(seq_lens, dtype=np.int64)) * w.g * w.d * 2 * 2


def run(args, w):
    import torch

    import paper_2406_09297_gb300 as mlkv
    from mlkv_synth import device, gen

    world, rank, local = _dist()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")

    cache = mlkv.MLKVCache(w.l, w.h, w.d, w.owner, w.g, w.b, w.max_seq)
    if args.tile:
        cache.set_option("tile_tokens", args.tile)
    if args.grid:
        cache.set_option("grid", args.grid)
    if args.cluster >= 0:
        cache.set_option("cluster", args.cluster)
    if args.l2_persist:
        cache.set_option("l2_persist", 1)
    if args.l2_prefetch >= 0:
        cache.set_option("l2_prefetch", args.l2_prefetch)
    if args.step_kernel >= 0:
        cache.set_option("step_kernel", args.step_kernel)
    if args.step_fused >= 0:
        cache.set_option("step_fused", args.step_fused)
    if args.fused_kc > 0:
        cache.set_option("fused_kc", args.fused_kc)
    if args.no_pdl:
        cache.set_option("pdl", 0)
    cache.set_option("tc", args.tc)
    owners = w.owners()
    seq_lens, Q, Kn, Vn = device.workload_inputs(w, cache)
    Qs = torch.stack(Q)                              # [l][b][h][d]
    Ks = torch.stack([Kn[n] for n in owners])        # [m][b][g][d], slot order
    Vs = torch.stack([Vn[n] for n in owners])
    outs = torch.empty((w.l, w.b, w.h, w.d), dtype=torch.bfloat16, device="cuda")
    out = list(outs.unbind(0))
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()

    def step():
        # one call: every layer in order, owner layers storing their new token and attending
        # in one launch; replayed from the CUDA graph the library recorded on the first call
        cache.decode_step(Qs, Ks, Vs, outs, seq_lens)

    step()
    cache.sync_status()
    step_info = {k: int(cache.get_option(k)) for k in ("last_step_kernel", "last_step_fused",
                                                        "last_step_launches", "last_fused_kc",
                                                        "last_grid", "last_tile_tokens",
                                                        "last_deferred_merge", "last_seg_major")}
    step_kernel = bool(step_info["last_step_kernel"])   # one launch for every layer
    fused = bool(step_info["last_step_fused"])          # ... in the cross-layer fused form
    # a decode launch per layer, or one for the whole step; each followed by a merge launch when
    # the split pieces' partials are merged after the decode (deferred merge); the fused form
    # stores the owners' new tokens in a launch of its own before its decode launch
    merges = 2 if cache.get_option("last_deferred_merge") else 1
    launches_per_step = (int(cache.get_option("last_step_launches")) if step_kernel
                         else merges * w.l)
    form = "fused" if fused else ("multi-layer" if step_kernel else "per-layer")

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()

    for _ in range(args.warmup):
        flush.zero_()
        step()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    barrier()
    with Clocks(local) as clocks:
        for k in range(args.steps):
            flush.zero_()
            ev[k][0].record()
            step()
            ev[k][1].record()
        barrier()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    ms = max_over_ranks(sum(step_ms) / len(step_ms), dist, "cuda")
    value = job_value(w.b, world, ms)
    spread = sorted(step_ms)   # the per-step times behind the mean, for the record

    # ---- the same step as a model runs it: one layer after another -----------------------------
    # A model computes layer n's queries from layer n-1's output, so its attention for layer n
    # reads nothing before layer n-1's has ended.  The step above is given every layer's queries
    # at once (the step call), which lets one launch cover every layer.  Here the same call runs
    # as one launch per layer (step_kernel 0) with no layer reading its queries before the
    # previous one has finished: in plain stream order (pdl 0), and with each grid's launch,
    # set-up and first cache tile overlapping the previous one's end, its queries read after it
    # (pdl 1, early_fetch 2: the cache and the owner's new token exist before the layer's queries
    # do).  L2 is flushed before each step as above.
    def time_with(options):
        saved = {k: int(cache.get_option(k)) for k in options}
        for key, val in options.items():
            cache.set_option(key, val)
        for _ in range(args.warmup):
            flush.zero_()
            step()
        sev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
        barrier()
        for k in range(args.steps):
            flush.zero_()
            sev[k][0].record()
            step()
            sev[k][1].record()
        barrier()
        t = max_over_ranks(sum(a.elapsed_time(b) for a, b in sev) / args.steps, dist, "cuda")
        n_launch = w.l * (2 if cache.get_option("last_deferred_merge") else 1)
        for key, val in saved.items():
            cache.set_option(key, val)
        return t, n_launch

    seq_ms, seq_launches = time_with({"step_kernel": 0, "pdl": 0})
    seqp_ms, _ = time_with({"step_kernel": 0, "pdl": 1, "early_fetch": 2})
    step()   # back to the measured configuration
    # ---- decode kernel durations ---------------------------------------------------------------
    # The graph-timed step is nothing but the l decode launches back to back, so its device time
    # divided by l is the mean launch duration inside the step.  Eager launches bracketed by events
    # (after a long flush, so the host queues ahead) give each layer's time, cold-L2 owner layers
    # apart from the layers that re-read a slot an earlier layer just streamed.
    big_flush = torch.empty(4 * FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    kev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in range(w.l)] for _ in range(args.steps)]
    torch.cuda.synchronize()
    for k in range(args.steps):
        big_flush.zero_()      # long enough for the host to queue the whole step behind it
        for n in range(w.l):
            kev[k][n][0].record()
            if n in Kn:
                cache.append_decode_attention(n, Kn[n], Vn[n], Q[n], out[n], seq_lens)
            else:
                cache.decode_attention(n, Q[n], out[n], seq_lens)
            kev[k][n][1].record()
    torch.cuda.synchronize()
    kms = [[a.elapsed_time(b) for a, b in row] for row in kev]
    layer_ms = [statistics.median(kms[k][n] for k in range(args.steps)) for n in range(w.l)]
    mean_kernel_ms = ms / w.l   # per layer; a merge launch, if any, is counted in with its decode
    kv_layer = kv_bytes_per_layer(w, seq_lens)
    qo_layer = 2 * w.b * w.h * w.d * 2
    alg_bytes = kv_layer + qo_layer
    peak, peak_kind = _peaks()
    achieved = alg_bytes / (mean_kernel_ms / 1e3) / 1e9
    # per launch: one layer, or every layer when the step is one multi-layer launch (the ratio
    # of bytes to time is the same)
    launch_bytes = alg_bytes * (w.l if step_kernel else 1)
    launch_ms = ms if step_kernel else mean_kernel_ms
    # The step's floor in DRAM bytes: every owner slot's visible rows once (the later layers of a
    # block could read them from L2), every layer's queries and outputs once.
    unique_bytes = len(w.owners()) * kv_layer + w.l * qo_layer
    unique_gbs = unique_bytes / (ms / 1e3) / 1e9
    cold = [layer_ms[n] for n in range(w.l) if w.owner[n] == n]
    cold_gbs = alg_bytes / (statistics.mean(cold) / 1e3) / 1e9
    del big_flush
    kernel_name = ("prefill_kernel" if fused else
                   "decode_tc_kernel" if cache.get_option("last_tc") else "decode_kernel")
    options = {k: int(cache.get_option(k)) for k in ("l2_prefetch", "l2_persist", "tc",
                                                      "step_kernel", "step_fused",
                                                      "l2_persist_bytes", "l2_window_max")}
    options.update(step_info)   # the measured step's launch, read right after its first call
    traffic = _recorded_traffic(w, kernel_name, form)

    # ---- end to end through the C ABI with host buffers --------------------------------------
    host_q = Qs.cpu().pin_memory()
    host_k = Ks.cpu().pin_memory()
    host_v = Vs.cpu().pin_memory()
    host_out = torch.empty((w.l, w.b, w.h, w.d), dtype=torch.bfloat16).pin_memory()
    h2d = (host_q.numel() + host_k.numel() + host_v.numel()) * 2
    d2h = host_out.numel() * 2

    def e2e_step():
        # the user's view: this step's inputs from pinned host memory, one library call for the
        # step, every layer's output back to pinned host memory
        mlkv.mlkv_decode_step_host(cache.handle, host_q, host_k, host_v, host_out, seq_lens)

    for _ in range(args.warmup):
        flush.zero_()
        e2e_step()
    torch.cuda.synchronize()
    e_times = []
    for _ in range(args.steps):
        # As for the device-timed steps, the L2 flush keeps the GPU busy while the host queues the
        # call (a user loop queues step k+1 while step k runs); the host then waits for this step's
        # outputs in host memory before the next.
        flush.zero_()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        e2e_step()
        e1.record()
        e1.synchronize()
        e_times.append(e0.elapsed_time(e1))
    e_ms = max_over_ranks(sum(e_times) / len(e_times), dist, "cuda")
    e2e_val = job_value(w.b, world, e_ms)
    cache.sync_status()

    result = None
    if rank == 0:
        result = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms,
            "step_ms": {"min": spread[0], "median": spread[len(spread) // 2], "max": spread[-1]},
            "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": _config_dict(w),
            "e2e": {"value": e2e_val, "unit": UNIT, "h2d_bytes_per_step": int(h2d),
                    "d2h_bytes_per_step": int(d2h), "ms_per_step": e_ms},
            "gpu_launches": launches_per_step * args.steps,
            "sequential_layers": {
                "value": job_value(w.b, world, seq_ms), "unit": UNIT, "ms_per_step": seq_ms,
                "launches_per_step": seq_launches,
                "overlapped_launch": {"value": job_value(w.b, world, seqp_ms),
                                      "ms_per_step": seqp_ms},
                "how": "the same step as one launch per layer, no layer reading its queries "
                       "before the previous one has finished, as in a model whose layer n "
                       "queries come from layer n-1: plain stream order (options step_kernel 0, "
                       "pdl 0); overlapped_launch: each grid's launch, set-up and first cache "
                       "tile overlap the previous one's end (step_kernel 0, pdl 1, early_fetch 2)"},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": traffic,
                         "peak_source": peak_kind,
                         "frac_vs_8tbs": achieved / 8000.0,
                         # achieved counts every layer's K/V (the per-layer reads the paper's
                         # implementation makes): "effective" once layers share a slot, since the
                         # step moves each owner slot from DRAM once (dram_frac_step; traffic)
                         "achieved_bytes": "logical K/V + Q + out of every layer (effective "
                                           "where layers share a slot)",
                         "kernel": kernel_name, "step_form": form,
                         "alg_bytes_per_launch": launch_bytes,
                         "mean_launch_ms": launch_ms, "launches_per_step": launches_per_step,
                         # the merge launch's time is inside mean_launch_ms (timed together),
                         # and in the fused form the new tokens' store launch's
                         "merge_time_included": merges == 2,
                         "append_time_included": fused,
                         "step_ms_per_layer": mean_kernel_ms,
                         "dram_unique_bytes_per_step": unique_bytes,
                         "dram_unique_gbs": unique_gbs,
                         "dram_frac_step": unique_gbs / peak,
                         "owner_launch_gbs": cold_gbs, "owner_launch_frac": cold_gbs / peak},
            "options": options,
            "step_kv_gbs": kv_layer * w.l / (ms / 1e3) / 1e9,
            "layer_ms": layer_ms,
            "clocks": clocks.summary(),
        }
        if world == 1 and not args.no_cpu_baseline:
            result["cpu_baseline"] = cpu_baseline(w)
    cache.close()
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return result


# The nine Pythia-160M variants of Table 2 (Sec. 4.2): (name, owner layers m, KV heads g), block map
# of Eq. 18.
TABLE2_VARIANTS = [("baseline", 12, 12), ("gqa-48", 12, 4), ("mlkv-48", 4, 12), ("mqa-12", 12, 1),
                   ("mlkv-12", 4, 3), ("mlkv-6", 6, 1), ("mlkv-4", 4, 1), ("mlkv-2", 2, 1),
                   ("mlkv-1", 1, 1)]
LOOP_PREFIX, LOOP_STEPS = 2000, 48


def run_loop(args):
    """The paper's throughput measurement (Sec. 4.5) on this library: a cache pre-filled with 2000
    positions, then 48 autoregressive decode steps -- every step appends a new token per owner
    layer (lengths grow by one) and attends in all 12 layers, one mlkv_decode_step call per step.
    Timed on the device over whole 48-step loops (host work between steps included, as it is in
    a decode loop), L2 flushed before each loop; tokens/s = batch * 48 / loop time, per variant.
    Attention only (the paper times the whole model)."""
    import torch

    import paper_2406_09297_gb300 as mlkv
    from mlkv_synth import device

    torch.cuda.set_device(0)
    l, h, d, b = 12, 12, 64, args.loop_batch
    max_seq = LOOP_PREFIX + LOOP_STEPS
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    results, per_step_us = {}, {}
    for name, m, g in TABLE2_VARIANTS:
        owner = [int(x) for x in mlkv.mlkv_block_owner_map(l, m)]
        owners = sorted(set(owner))
        seed = 2000 + m * 16 + g
        with mlkv.MLKVCache(l, h, d, owner, g, b, max_seq) as cache:
            cache.set_option("tc", args.tc)
            if args.grid:
                cache.set_option("grid", args.grid)
            if args.cluster >= 0:
                cache.set_option("cluster", args.cluster)
            if args.step_fused >= 0:
                cache.set_option("step_fused", args.step_fused)
            if args.fused_kc > 0:
                cache.set_option("fused_kc", args.fused_kc)
            for n in owners:
                kp, vp, strides = cache.kv_ptr(cache.owner_slot(n)[1])
                device.fill_slot(kp, vp, strides, seed, n, b, g, d, max_seq)
            lens = [np.full(b, LOOP_PREFIX + s + 1, dtype=np.int32) for s in range(LOOP_STEPS)]
            # per step: every layer's queries (another seed per step) and every owner's new token
            Qs = [torch.stack([device.q_tensor(seed + 1 + s, n, b, h, d) for n in range(l)])
                  for s in range(LOOP_STEPS)]
            Ks = [torch.stack([device.kv_token(seed, n, 0, b, g, d, lens[s]) for n in owners])
                  for s in range(LOOP_STEPS)]
            Vs = [torch.stack([device.kv_token(seed, n, 1, b, g, d, lens[s]) for n in owners])
                  for s in range(LOOP_STEPS)]
            out = torch.empty((l, b, h, d), dtype=torch.bfloat16, device="cuda")

            def loop():
                for s in range(LOOP_STEPS):
                    cache.decode_step(Qs[s], Ks[s], Vs[s], out, lens[s])

            for _ in range(max(args.warmup, 1)):
                loop()
            cache.sync_status()
            times = []
            for _ in range(args.loop_reps):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                loop()
                e1.record()
                torch.cuda.synchronize()
                times.append(e0.elapsed_time(e1))
            cache.sync_status()
            ms = statistics.median(times)
            results[name] = b * LOOP_STEPS / (ms / 1e3)
            per_step_us[name] = ms * 1e3 / LOOP_STEPS
    line = {"metric": "decode-loop tokens/s (prefix 2000, 48 decode steps, attention only)",
            "unit": "tokens/s", "higher_is_better": True, "batch": b, "layers": l, "q_heads": h,
            "head_dim": d, "reps": args.loop_reps, "dtype": "bf16", "data": "synthetic",
            "kernel": "decode_tc_kernel" if args.tc else "decode_kernel",
            "results": {k: round(v, 1) for k, v in results.items()},
            "us_per_step": {k: round(v, 2) for k, v in per_step_us.items()}}
    print(json.dumps(line), flush=True)


def _tensor_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def run_prefill(args, w):
    """Prefill of a whole prompt per sequence through every layer of the workload's model, in layer
    order (owner layers store the prompt's K/V, every layer attends causally over its owner's
    slot): one mlkv_prefill per layer, timed on the device, L2 flushed before each repetition.
    tokens/s = batch * prompt / time; TFLOP/s counts the useful causal work
    4 * h * d * sum_beta S (S + 1) / 2 per layer (QK^T and PV, 2 flops a multiply-add)."""
    import torch

    import paper_2406_09297_gb300 as mlkv
    from mlkv_synth import device

    torch.cuda.set_device(0)
    b, S = args.prefill_batch, args.prefill_len
    owners = w.owners()
    with mlkv.MLKVCache(w.l, w.h, w.d, w.owner, w.g, b, S) as cache:
        Q = [torch.empty((b, S, w.h, w.d), dtype=torch.bfloat16, device="cuda") for _ in range(w.l)]
        for n in range(w.l):
            device.fill_(Q[n].view(b * S, w.h * w.d), w.seed + 1, 0x100 + n, w.sigma_q)
        KV = {}
        for n in owners:
            k = torch.empty((b, w.g, S, w.d), dtype=torch.bfloat16, device="cuda")
            v = torch.empty_like(k)
            device.fill_(k.view(b * w.g, S * w.d), w.seed + 1, 0x200 + n, w.sigma_k)
            device.fill_(v.view(b * w.g, S * w.d), w.seed + 1, 0x300 + n, w.sigma_v)
            KV[n] = (k, v)
        out = torch.empty((b, S, w.h, w.d), dtype=torch.bfloat16, device="cuda")
        lens = np.full(b, S, dtype=np.int32)
        flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")

        def prefill_model():
            for n in range(w.l):
                k, v = KV.get(n, (None, None))
                cache.prefill(n, Q[n], k, v, out, lens)

        for _ in range(args.warmup):
            prefill_model()
        cache.sync_status()
        times = []
        with Clocks(0) as clocks:
            for _ in range(args.steps):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                prefill_model()
                e1.record()
                torch.cuda.synchronize()
                times.append(e0.elapsed_time(e1))
        cache.sync_status()
    ms = statistics.median(times)
    flops = 4.0 * w.h * w.d * b * S * (S + 1) / 2 * w.l
    tflops = flops / (ms / 1e3) / 1e12
    peak, kind = _tensor_peak()
    line = {"metric": "prefill tokens/s (all layers, causal)", "value": b * S / (ms / 1e3),
            "unit": "tokens/s", "higher_is_better": True, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name, "layers": w.l, "q_heads": w.h, "head_dim": w.d,
                       "layer_owner": list(w.owner), "kv_heads_per_owner": w.g, "batch": b,
                       "prompt": S, "l2": "flushed before every timed repetition"},
            "roofline": {"bound": "tensor", "achieved": tflops, "peak": peak, "unit": "TFLOP/s",
                         "frac": tflops / peak, "peak_source": kind, "kernel": "prefill_kernel",
                         "flops_per_step": flops},
            "clocks": clocks.summary()}
    print(json.dumps(line), flush=True)


def _hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def run_l2_peak(args):
    """Read bandwidth of L2-resident data, the roofline of a decode layer whose owner slot an
    earlier layer of its block has just brought into L2 (a Pythia-160M MLKV-2 slot at batch 64,
    context 2048 is 32 MiB): the library's read-bandwidth probe (bulk copies into a shared-memory
    ring, as the decode kernel moves K/V) over a 32 MiB and a 64 MiB buffer, 20 passes in one
    launch, and over a 4 GiB buffer (HBM), CUDA events around each launch, best of five."""
    import torch

    import paper_2406_09297_gb300 as mlkv
    torch.cuda.set_device(0)
    res = {}
    for name, nbytes, reps in (("l2_32MiB", 32 << 20, 20), ("l2_64MiB", 64 << 20, 20),
                               ("hbm_4GiB", 4 << 30, 1)):
        buf = torch.ones(nbytes // 2, dtype=torch.bfloat16, device="cuda")
        best = 0.0
        for _ in range(6):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            n = mlkv.mlkv_read_bandwidth_probe(buf, reps)
            e1.record()
            e1.synchronize()
            best = max(best, n / (e0.elapsed_time(e1) / 1e3) / 1e9)
        res[name + "_gbs"] = best
        del buf
    line = {"metric": "read bandwidth (bulk copies into shared memory)", "unit": "GB/s", **res,
            "hbm_copy_gbs_measured_peaks": _hbm_peak()[0],
            "how": "mlkv_read_bandwidth_probe: 2 CTAs per SM, 32 KiB copies, 2-stage ring; "
                   "CUDA events around one launch; best of 6 (first one warms L2)"}
    print(json.dumps(line), flush=True)


def run_merge(args, w):
    """Sec. 4.2 conversion of the workload's model: its MHA K and V projections (l x h heads, each
    head_dim x d_model, d_model = h * head_dim, seeded bf16) merged by averaging into the owner
    map's m x g KV heads.  Both projections go through one mlkv_merge_kv_weights call: stacked as
    2 l layers, K's then V's, with V's layers owned by owner + l, the merged heads come out K's
    then V's (the merge never mixes layers of different owners).  L2 flushed before each
    repetition.  HBM-bound: algorithmic bytes = inputs read once + outputs written once."""
    import torch

    import paper_2406_09297_gb300 as mlkv
    from mlkv_synth import device, gen

    torch.cuda.set_device(0)
    row = w.d * w.h * w.d
    m = len(w.owners())
    W = torch.empty((2, w.l, w.h, row), dtype=torch.bfloat16, device="cuda")
    for kv in range(2):
        for n in range(w.l):
            device.fill_(W[kv, n], w.seed + 7, gen.TID_W + 64 * kv + n, 0.02)
    out = torch.empty((2, m, w.g, row), dtype=torch.bfloat16, device="cuda")
    owner2 = list(w.owner) + [o + w.l for o in w.owner]
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()

    def step():
        mlkv.mlkv_merge_kv_weights(owner2, w.h, w.g, W.view(2 * w.l, w.h, row),
                                   out.view(2 * m, w.g, row), stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    times = []
    with Clocks(0) as clocks:
        for _ in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            step()
            e1.record(stream)
            torch.cuda.synchronize()
            times.append(e0.elapsed_time(e1))
    ms = statistics.median(times)
    nbytes = 2 * 2 * (w.l * w.h + m * w.g) * row
    gbs = nbytes / (ms / 1e3) / 1e9
    peak, kind = _hbm_peak()
    line = {"metric": "KV-weight merge GB/s (K and V projections)", "value": gbs, "unit": "GB/s",
            "higher_is_better": True, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name, "layers": w.l, "q_heads": w.h, "head_dim": w.d,
                       "d_model": w.h * w.d, "layer_owner": list(w.owner), "kv_heads_per_owner": w.g,
                       "l2": "flushed before every timed repetition"},
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peak, "unit": "GB/s",
                         "frac": gbs / peak, "peak_source": kind, "kernel": "merge_kernel",
                         "alg_bytes_per_step": nbytes, "launches_per_step": 1},
            "clocks": clocks.summary()}
    print(json.dumps(line), flush=True)


def run_fused(args, w):
    """Cross-layer fused decode (benchmark only: a model never has every layer's queries at once):
    one step = for every owner, its new token appended and all its block's layers decoded in one
    mlkv_decode_block_fused launch, which reads each K/V tile of the slot once.  Same inputs and
    tokens/s as the decode step of run(); L2 flushed before every step."""
    import torch

    import paper_2406_09297_gb300 as mlkv
    from mlkv_synth import device

    torch.cuda.set_device(0)
    owners = w.owners()
    cache = mlkv.MLKVCache(w.l, w.h, w.d, w.owner, w.g, w.b, w.max_seq)
    seq_lens, Q, Kn, Vn = device.workload_inputs(w, cache)
    blocks = {o: [n for n in range(w.l) if w.owner[n] == o] for o in owners}
    Qb = {o: torch.stack([Q[n] for n in blocks[o]]) for o in owners}
    outs = {o: torch.empty_like(Qb[o]) for o in owners}
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()

    def step():
        for o in owners:
            cache.append(o, Kn[o], Vn[o], seq_lens, stream)
            cache.decode_block_fused(o, Qb[o], outs[o], seq_lens, stream)

    for _ in range(args.warmup):
        step()
    cache.sync_status()
    times = []
    with Clocks(0) as clocks:
        for _ in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            step()
            e1.record(stream)
            torch.cuda.synchronize()
            times.append(e0.elapsed_time(e1))
    cache.sync_status()
    ms = statistics.median(times)
    tot_len = int(np.sum(seq_lens))
    kv_bytes = 2 * len(owners) * w.g * tot_len * w.d * 2          # every slot read once
    qo_bytes = 2 * w.l * w.b * w.h * w.d * 2
    gbs = (kv_bytes + qo_bytes) / (ms / 1e3) / 1e9
    flops = 4.0 * w.h * w.d * tot_len * w.l
    peak, kind = _hbm_peak()
    line = {"metric": "decode-attn tokens/s per step (all layers), cross-layer fused",
            "value": w.b / (ms / 1e3), "unit": "tokens/s", "higher_is_better": True,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "dtype": "bf16",
            "data": "synthetic", "benchmark_only": "needs every layer's queries at once",
            "config": {"workload": w.name, "layers": w.l, "q_heads": w.h, "head_dim": w.d,
                       "layer_owner": list(w.owner), "kv_heads_per_owner": w.g, "batch": w.b,
                       "context": w.L, "l2": "flushed before every timed step"},
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peak, "unit": "GB/s",
                         "frac": gbs / peak, "peak_source": kind, "kernel": "prefill_kernel (fused)",
                         "alg_bytes_per_step": kv_bytes + qo_bytes,
                         "tensor_tflops_useful": flops / (ms / 1e3) / 1e12},
            "gpu_launches": 2 * len(owners), "clocks": clocks.summary()}
    print(json.dumps(line), flush=True)
    cache.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--config", default=DEFAULT_WORKLOAD)
    ap.add_argument("--tile", type=int, default=0)
    ap.add_argument("--grid", type=int, default=0)
    ap.add_argument("--cluster", type=int, default=-1, choices=[-1, 0, 1, 2, 4],
                    help="decode 'cluster' option (-1: the library default)")
    ap.add_argument("--l2-persist", action="store_true")
    ap.add_argument("--l2-prefetch", type=int, default=-1, choices=[-1, 0, 1],
                    help="option l2_prefetch (-1: the library's default)")
    ap.add_argument("--step-kernel", type=int, default=-1, choices=[-1, 0, 1],
                    help="option step_kernel (-1: the library's default)")
    ap.add_argument("--step-fused", type=int, default=-1, choices=[-1, 0, 1, 2],
                    help="option step_fused (-1: the library's default)")
    ap.add_argument("--fused-kc", type=int, default=0,
                    help="option fused_kc: key tiles per unit of the fused step (0: planned)")
    ap.add_argument("--no-pdl", action="store_true")
    ap.add_argument("--tc", type=int, default=0, choices=[0, 1],
                    help="0: the mma.sync decode kernel (default); 1: the tcgen05 kernel")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--loop", action="store_true",
                    help="the decode-loop measurement over the nine Table 2 variants")
    ap.add_argument("--loop-batch", type=int, default=8)
    ap.add_argument("--loop-reps", type=int, default=5)
    ap.add_argument("--prefill", action="store_true",
                    help="prefill throughput of the --config model (prompt of --prefill-len)")
    ap.add_argument("--prefill-batch", type=int, default=8)
    ap.add_argument("--prefill-len", type=int, default=2048)
    ap.add_argument("--fused", action="store_true",
                    help="cross-layer fused decode of the --config workload (benchmark only)")
    ap.add_argument("--l2-peak", action="store_true",
                    help="measure the read bandwidth of an L2-resident buffer")
    ap.add_argument("--merge", action="store_true",
                    help="Sec. 4.2 KV-weight merge of the --config model's K and V projections")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.loop:
        run_loop(args)
        return
    if args.prefill:
        from mlkv_synth import workloads
        run_prefill(args, workloads.by_name(args.config))
        return
    if args.l2_peak:
        run_l2_peak(args)
        return
    if args.merge:
        from mlkv_synth import workloads
        run_merge(args, workloads.by_name(args.config))
        return
    if args.fused:
        from mlkv_synth import workloads
        run_fused(args, workloads.by_name(args.config))
        return

    from mlkv_synth import workloads
    w = workloads.by_name(args.config)
    if args.impl == "reference":
        run_reference(args, w)
        return
    res = run(args, w)
    if res is not None:
        print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
