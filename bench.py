"""Benchmark of the PRCR revisit path (rebind + inject) on GB300.

One step = one call of the public entry point prcr_rebind_inject over one
batch: the plan kernel (positions, slots) and the fused gather / M-RoPE
rebind / inject kernel (one kernel for small batches), for every selected
token x layer x KV head of every sequence in the batch.

Default workload: the largest one (16-frame 16x32x32 video per sequence,
4096 revisited tokens per sequence in 3 revisits, batch 32, 36 layers, 8 KV
heads, head_dim 128, paged cache with block 16): 38.65 GB moved per step,
far larger than L2, so no flush is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle on bounded samples

Prints one JSON line (rank 0). Under torchrun (N > 1) every rank runs its own
full batch on its own GPU (weak scaling, no collective on the data path);
the step time is the maximum over ranks.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)
# the oracle legs run on one host thread (their `cores`): numpy's BLAS and
# OpenMP pools are fixed before anything imports numpy
for _v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")

METRIC = "rebind+inject GB/s (read+write)"
UNIT = "GB/s"
SPEC_HBM_GBS = 8000.0

# DRAM traffic (read + write bytes) of one rebind launch on the default
# workload, from an ncu capture; valid only for the kernel source it was
# measured on (its sha256 prefix), reported as null otherwise.
TRAFFIC = {
    # captured on the stress shape cut to 2 sequences (8,192 tokens: 1,193,440,000 B
    # read + 1,150,144,256 B written) and scaled by the 16x more tokens of a full launch
    ("stress", "46dd442ca336fc40"): 37497348096,
}

# the Table 3 shapes (Qwen3-VL-8B dimensions, a 768-token image, K = 32 and
# K = 128), timed after the main workload
PAPER_SHAPES = ("paper-8b-k32", "paper-8b-k128")


def _sha(*paths):
    """Hash of the rebind kernel's sources: a stored traffic figure is used
    only while they are the ones it was measured on."""
    h = hashlib.sha256()
    for path in paths:
        with open(path, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["prcr", "reference"], default="prcr")
    ap.add_argument("--workload", default="stress")
    ap.add_argument("--path", choices=["revisit", "capture", "decode", "select", "pipeline"],
                    default="revisit",
                    help="revisit: the rebind+inject step (default); capture: prefill capture; "
                         "decode: the first decode step over the active cache; select: the "
                         "attention-driven selection of the revisited set; pipeline: select, "
                         "rebind+inject and the first decode step of one revisit, end to end")
    ap.add_argument("--seqs", type=int, default=0,
                    help="sequences of the workload's batch (0 = the workload's own count)")
    ap.add_argument("--select-source", choices=["raw", "cache"], default="raw",
                    help="select / pipeline: rank from the raw store (prcr_select_topk) or from "
                         "the position-bound cache (prcr_select_topk_cached)")
    ap.add_argument("--max-len", type=int, default=8192,
                    help="decode: the longest sequence (lengths drawn in [1, max-len], the last "
                         "one at max-len)")
    ap.add_argument("--layers", type=int, default=0,
                    help="select: build the store with this many layers (0 = workload's); "
                         "the selection reads the last one")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-samples", type=int, default=8,
                    help="sequences the CPU oracle baseline is timed on")
    ap.add_argument("--no-check", action="store_true", help="skip the pre-timing parity check")
    ap.add_argument("--graph", action="store_true",
                    help="replay the step from a CUDA graph (for small, launch-bound workloads)")
    ap.add_argument("--graph-inner", type=int, default=20, help="steps captured per graph")
    ap.add_argument("--flush", choices=["auto", "on", "off"], default="auto",
                    help="write a buffer of twice the L2 size before each timed step "
                         "(auto: when a step moves less than 4x the L2 size)")
    ap.add_argument("--no-paper-shape", action="store_true",
                    help="skip the Table 3 shape latencies of the revisit path")
    ap.add_argument("--no-next-rows", action="store_true",
                    help="skip the NEXT rows' numbers (selection, small-batch decode, one "
                         "revisit end to end) in the revisit path's line")
    return ap.parse_args()


def kernel_launches(fn):
    """Names, in launch order, of this library's CUDA kernels one call of fn
    launches, as the profiler (CUPTI) records them; empty if it records none.
    (Kernel records come only with CPU activity profiled too.)"""
    import re
    import torch
    from torch.profiler import ProfilerActivity, profile
    torch.cuda.synchronize()
    for _ in range(3):  # the first session of a process records no kernels
        with profile(activities=[ProfilerActivity.CPU, ProfilerActivity.CUDA]) as prof:
            fn()
            torch.cuda.synchronize()
        evs = sorted((e for e in prof.events() if e.device_type.name == "CUDA"),
                     key=lambda e: e.time_range.start)
        out = []
        for e in evs:
            m = re.search(r"\bprcr::.*?\b(\w+_kernel)\b", e.name)
            if m:
                out.append(m.group(1))
        if out:
            return out
    return []


class L2Flush:
    """Evicts L2 between timed steps: writes a buffer of twice its size, then
    reads another of twice its size, so that the next step finds none of its
    inputs in L2 and no dirty lines whose write-back would land inside its
    timed region (a write alone leaves ~one L2 of dirty lines behind)."""

    def __init__(self, dev, mode, nbytes):
        import torch
        self.l2 = int(getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 0)) or (129 << 20)
        self.enabled = mode == "on" or (mode == "auto" and nbytes < 4 * self.l2)
        self.buf = torch.empty(2 * self.l2, dtype=torch.uint8, device=dev) if self.enabled else None
        self.rbuf = (torch.zeros(2 * self.l2 // 4, dtype=torch.int32, device=dev)
                     if self.enabled else None)
        self.sink = torch.zeros((), dtype=torch.int64, device=dev) if self.enabled else None
        self.i = 0

    def __call__(self):
        if self.enabled:
            self.i += 1
            self.buf.fill_(self.i & 0xFF)
            self.sink.add_(self.rbuf.sum())

    def describe(self, nbytes):
        if self.enabled:
            return ("L2 flushed before each step (%d MB written, then %d MB of another buffer "
                    "read); each step moves %.2f GB" % (2 * self.l2 >> 20, 2 * self.l2 >> 20,
                                                      nbytes / 1e9))
        if nbytes >= 4 * self.l2:
            return "inputs larger than L2 (no flush): each step moves %.2f GB" % (nbytes / 1e9)
        return ("warm: no flush between steps, %.2f GB per step against a %d MB L2"
                % (nbytes / 1e9, self.l2 >> 20))


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(value: float, world: int, device=None) -> float:
    """Maximum of a per-rank float over all ranks (identity at world 1)."""
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ----------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------
class Clocks:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-f", self.path], stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        pw = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows), "power_w_max": max(pw) if pw else None}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ----------------------------------------------------------------------------
# the CPU oracle on a bounded sample
# ----------------------------------------------------------------------------
def sample_batch(wl, n_layers: int, n_tokens=None, device="cpu", seed: int = 0):
    """A bounded sample of the workload: its first sequence (same grids,
    selection recipe and value distribution) with n_layers layers, optionally
    cut to the first n_tokens selected tokens (one revisit), on the host."""
    from workloads import make_batch
    import torch
    b = make_batch(dataclasses.replace(wl, n_seqs=1, n_layers=n_layers), device=device, seed=seed)
    if device != "cpu":
        b = dataclasses.replace(b, **{f: getattr(b, f).cpu() for f in (
            "store_k", "store_v", "coords", "seq_rev_off", "rev_tok_off", "idx", "p_txt",
            "cache_len_in")})
    if n_tokens is not None and n_tokens < b.total_k:
        b = dataclasses.replace(b, idx=b.idx[:n_tokens].clone(),
                                rev_tok_off=torch.tensor([0, n_tokens], dtype=torch.int32),
                                seq_rev_off=torch.tensor([0, 1], dtype=torch.int32))
    return b


def oracle_step(batch):
    """Time the oracle's whole call on the batch (positions, gather, rebind,
    value copy) on the host; returns seconds."""
    import numpy as np
    import torch
    from oracle import prcr_oracle as O
    wl = batch.wl
    kb = batch.store_k.view(torch.int16).numpy()
    vb = batch.store_v.view(torch.int16).numpy()
    t0 = time.perf_counter()
    out = O.rebind_inject(kb, vb, batch.coords.numpy(), batch.seq_rev_off.numpy(),
                          batch.rev_tok_off.numpy(), batch.idx.numpy(), batch.p_txt.numpy(),
                          batch.cache_len_in.numpy(), wl.head_dim, wl.sections, wl.theta, wl.L)
    dt = time.perf_counter() - t0
    assert np.isfinite(out["k_hat"]).all()
    return dt


def describe_sample(wl, batch):
    return (f"sequence 0 of '{wl.name}': {batch.total_k} selected tokens in {batch.n_revisits} "
            f"revisit(s) x {batch.wl.n_layers} of {wl.n_layers} layers x {wl.n_kv_heads} KV heads "
            f"({batch.algorithmic_bytes() / 1e6:.1f} MB algorithmic); numpy float64, one thread")


def cpu_baseline(wl, n_layers: int, n_samples: int = 1, device="cpu"):
    """The oracle's whole call timed on n_samples sequences drawn like the
    workload's (seeds 0 .. n_samples-1), one sequence per call."""
    total_t, total_b, batch = 0.0, 0, None
    for s in range(n_samples):
        batch = sample_batch(wl, n_layers, device=device, seed=s)
        total_t += oracle_step(batch)
        total_b += batch.algorithmic_bytes()
        del batch
    return dict(value=total_b / total_t / 1e9, unit=UNIT, cores=1, host_cores=os.cpu_count(),
                kind="oracle",
                sample=(f"{n_samples} sequence(s) drawn like '{wl.name}' (seeds 0..{n_samples - 1}), "
                        f"all selected tokens x {n_layers} of {wl.n_layers} layers x "
                        f"{wl.n_kv_heads} KV heads, one sequence per oracle call "
                        f"({total_b / 1e9:.2f} GB algorithmic); numpy float64, one thread"),
                seconds=total_t)


def oracle_leg(args, fn, nbytes: int, sample: str):
    """The oracle as it stands, timed once on the host on a bounded sample of
    the path's workload: GB/s of the sample's algorithmic bytes."""
    if args.no_cpu_baseline:
        return None
    t0 = time.perf_counter()
    fn()
    dt = time.perf_counter() - t0
    return dict(value=nbytes / dt / 1e9, unit=UNIT, cores=1, host_cores=os.cpu_count(),
                kind="oracle", sample=sample + "; numpy float64, one thread", seconds=dt)


# ----------------------------------------------------------------------------
# reference arm: the oracle as it stands, timed on the host cores
# ----------------------------------------------------------------------------
REF_TOKENS = 512  # tokens of one revisit, one layer, per reference step


def run_reference(args):
    world, rank, local = dist_env()
    if rank != 0:
        return
    from workloads import get
    wl = get(args.workload)
    batch = sample_batch(wl, 1, n_tokens=REF_TOKENS)
    for _ in range(args.warmup):
        oracle_step(batch)
    times = [oracle_step(batch) for _ in range(args.steps)]
    t = sum(times)
    nbytes = batch.algorithmic_bytes() * args.steps
    value = nbytes / t / 1e9
    line = dict(metric=METRIC, value=value, unit=UNIT, n_gpus=args.gpus, steps=args.steps,
                warmup=args.warmup, ms_per_step=1e3 * t / args.steps, higher_is_better=True,
                scaling="weak", vs_baseline=None, dtype="f64", data="synthetic",
                config=dict(workload=wl.name, sample_per_step=describe_sample(wl, batch)),
                impl="reference",
                cpu_baseline=dict(kind="oracle", cores=1, host_cores=os.cpu_count(), value=value,
                                  unit=UNIT, sample=describe_sample(wl, batch)),
                e2e=dict(value=value, unit=UNIT, h2d_bytes_per_step=0, d2h_bytes_per_step=0),
                gpu_launches=0)
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------
def selection_manifest(wl, seed: int):
    """The JSON manifest of the revisits this rank's batch selects (drawn on
    the host by the workload generator), and whether it equals the committed
    copy under workloads/manifests/."""
    from workloads import manifest as MF
    m = MF.manifest(wl, seed)
    text = MF.dumps(m)
    path = MF.path_for(wl.name, seed)
    committed = os.path.exists(path) and open(path).read() == text
    return dict(path=os.path.relpath(path, ROOT) if committed else None,
                sha256=MF.sha256_of(text), matches_committed=committed,
                n_revisits=m["n_revisits"], total_k=m["total_k"])


def paper_shape_latency(dev, local, cold_steps: int = 100, inner: int = 20, replays: int = 10):
    """The revisit of Table 3's shapes (Qwen3-VL-8B dimensions, a 768-token
    image, one rectangle of K = 32 or 128 tokens, contiguous cache) through
    the public call prcr_rebind_inject: every output first compared with the
    oracle; then `cold` = stream launches each after a write of twice the L2
    size (the raw rows, plan inputs and cache lines not in L2), and `warm` =
    CUDA-graph replays of `inner` calls back to back (launch overhead gone,
    working set in L2). Microseconds per call."""
    import torch
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import parity_util as pu
    from workloads import get, make_batch
    out = {}
    stream = torch.cuda.current_stream()
    for name in PAPER_SHAPES:
        batch = make_batch(get(name), device=dev)
        rv = pu.make_revisit(batch)
        rv.run()
        torch.cuda.synchronize()
        if rv.status_value() != 0:
            raise RuntimeError(f"{name}: device status {rv.status_value():#x}")
        err = pu.full_check(batch, rv)
        launched = kernel_launches(rv.run)
        nbytes = batch.algorithmic_bytes()
        flush = L2Flush(dev, "on", nbytes)
        for _ in range(3):
            flush()
            rv.run()
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(cold_steps)]
        with Clocks(local) as clk:
            for e0, e1 in ev:
                flush()
                e0.record(stream)
                rv.run()
                e1.record(stream)
            torch.cuda.synchronize()
            cold = [1e3 * e0.elapsed_time(e1) for e0, e1 in ev]
            g = torch.cuda.CUDAGraph()
            side = torch.cuda.Stream()
            side.wait_stream(stream)
            with torch.cuda.stream(side):
                rv.run()
            stream.wait_stream(side)
            torch.cuda.synchronize()
            with torch.cuda.graph(g):
                for _ in range(inner):
                    rv.run()
            for _ in range(3):
                g.replay()
            torch.cuda.synchronize()
            evg = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(replays)]
            for e0, e1 in evg:
                e0.record(stream)
                g.replay()
                e1.record(stream)
            torch.cuda.synchronize()
            warm = [1e3 * e0.elapsed_time(e1) / inner for e0, e1 in evg]
        out[name] = dict(
            tokens=batch.total_k, bytes=nbytes, kernels=launched or None,
            cold_us_median=statistics.median(cold), cold_us_mean=statistics.mean(cold),
            warm_us_median=statistics.median(warm), warm_us_mean=statistics.mean(warm),
            cold_gbs=nbytes / statistics.median(cold) / 1e3,
            warm_gbs=nbytes / statistics.median(warm) / 1e3,
            cold_steps=cold_steps, warm_calls=inner * replays,
            l2=flush.describe(nbytes) + " (cold); no flush, graph replays (warm)",
            parity=dict(k_max_err=err["max_err"], positions_slots_v="bit-exact"),
            clocks=clk.summary())
        del rv, batch, g
        torch.cuda.empty_cache()
    return out


def run_gpu(args):
    import torch
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)

    from paper_2606_26631_gb300 import _build
    if not _build.up_to_date():
        if rank == 0:
            _build.build()
        barrier(world)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import parity_util as pu
    from workloads import get, make_batch

    wl = get(args.workload)
    if args.seqs:
        wl = dataclasses.replace(wl, n_seqs=args.seqs)
    batch = make_batch(wl, device=dev, seed=rank)
    rv = pu.make_revisit(batch)
    nbytes = batch.algorithmic_bytes()

    # correctness gate before timing: positions/slots everywhere, rows on samples
    rv.run()
    torch.cuda.synchronize()
    if rv.status_value() != 0:
        raise RuntimeError(f"device status {rv.status_value():#x}")
    check = None
    if not args.no_check:
        pl = pu.oracle_plan(batch)
        pu.check_plan(rv, pl)
        import numpy as np
        seqs = sorted({0, wl.n_seqs // 2, wl.n_seqs - 1})
        toks = np.nonzero(np.isin(pl["seq"], np.asarray(seqs)))[0]
        layers = sorted({0, wl.n_layers // 2, wl.n_layers - 1})
        e = pu.check_rows(batch, rv, pl, toks, layers)
        check = dict(k_max_err=e["max_err"], k_max_rel=e["max_rel"], rows_checked=e["n"],
                     positions_slots_bit_exact=True, v_bit_exact=True)

    stream = torch.cuda.current_stream()
    # what one public call launches: one fused kernel for small batches, or
    # the plan kernel then the rebind + inject kernel
    launched = kernel_launches(rv.run)
    split = launched == ["plan_kernel", "rebind_kernel"] or not launched
    per_step = len(launched) if launched else 2
    for _ in range(args.warmup):
        rv.run()
    torch.cuda.synchronize()
    flush = L2Flush(dev, "off" if args.graph else args.flush, nbytes)

    K = args.steps
    apply_ms = plan_ms = None
    if args.graph:
        # K steps as K / inner replays of a graph holding `inner` steps
        inner = max(1, args.graph_inner)
        K = max(inner, (K + inner - 1) // inner * inner)
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            rv.run()
        stream.wait_stream(side)
        torch.cuda.synchronize()
        with torch.cuda.graph(g):
            for _ in range(inner):
                rv.run()
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(K // inner)]
        barrier(world)
        torch.cuda.synchronize()
        with Clocks(local) as clk:
            for e0, e2 in ev:
                e0.record(stream)
                g.replay()
                e2.record(stream)
            torch.cuda.synchronize()
        barrier(world)
        step_ms = [e0.elapsed_time(e2) / inner for e0, e2 in ev for _ in range(inner)]
    else:
        # the headline: the public call, events around each step
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(K)]
        barrier(world)
        torch.cuda.synchronize()
        with Clocks(local) as clk:
            for e0, e2 in ev:
                flush()
                e0.record(stream)
                rv.run()
                e2.record(stream)
            torch.cuda.synchronize()
        barrier(world)
        step_ms = [e0.elapsed_time(e2) for e0, e2 in ev]
        # per-kernel durations for the roofline: the same work through the
        # call's two halves (prcr_plan, prcr_rebind_apply) with an event
        # between them, after the headline loop
        if split:
            R = min(K, 20)
            evk = [tuple(torch.cuda.Event(enable_timing=True) for _ in range(3)) for _ in range(R)]
            torch.cuda.synchronize()
            for e0, e1, e2 in evk:
                flush()
                e0.record(stream)
                rv.run_plan()
                e1.record(stream)
                rv.run_apply()
                e2.record(stream)
            torch.cuda.synchronize()
            apply_ms = [e1.elapsed_time(e2) for _, e1, e2 in evk]
            plan_ms = [e0.elapsed_time(e1) for e0, e1, _ in evk]
        else:
            apply_ms = step_ms
    total_s = sum(step_ms) / 1e3
    total_s = max_over_ranks(total_s, world, dev)
    value = nbytes * world * K / total_s / 1e9
    ms_per_step = 1e3 * total_s / K

    # end to end through the public call, host buffers, copies inside the timed region
    for _ in range(2):
        rv.run_from_host()
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(args.e2e_steps):
        st = rv.run_from_host()
        if st != 0:
            raise RuntimeError(f"device status {st:#x}")
    e2e_s = max_over_ranks(time.perf_counter() - t0, world, dev)
    e2e_value = nbytes * world * args.e2e_steps / e2e_s / 1e9

    peak, peak_kind = measured_peaks()
    if apply_ms is not None:
        apply_avg_s = statistics.mean(apply_ms) / 1e3
        kernel = "rebind_kernel" if split else "fused_kernel"
    else:  # graph replay: only whole steps are timed
        apply_avg_s = statistics.mean(step_ms) / 1e3
        kernel = " + ".join(launched or ["plan_kernel", "rebind_kernel"]) + " (graph step)"
    manifest = selection_manifest(wl, rank)
    shapes = None
    if rank == 0 and not args.no_paper_shape:
        shapes = paper_shape_latency(dev, local)
    achieved = nbytes / apply_avg_s / 1e9
    src_sha = _sha(*(os.path.join(ROOT, "paper_2606_26631_gb300", "csrc", f)
                     for f in ("prcr_rebind.cu", "prcr_device.cuh", "prcr_internal.h")))
    traffic = TRAFFIC.get((wl.name, src_sha)) if split else None
    roof = dict(bound="hbm", achieved=achieved, peak=peak, unit="GB/s", frac=achieved / peak,
                traffic=traffic, kernel=kernel, peak_kind=f"{peak_kind} copy (hbm_gbs)",
                bytes_per_launch=nbytes, avg_launch_us=1e6 * apply_avg_s)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(wl, wl.n_layers, n_samples=args.cpu_samples, device=dev)
    rows = None
    if rank == 0 and world == 1 and not args.no_next_rows:
        rows = next_rows(args)

    if rank == 0:
        R = batch.n_revisits
        line = dict(
            metric=METRIC, value=value, unit=UNIT, n_gpus=world, steps=K, warmup=args.warmup,
            ms_per_step=ms_per_step, higher_is_better=True, scaling="weak", vs_baseline=None,
            dtype="f32", io_dtype="bf16", data="synthetic",
            config=dict(workload=wl.name, n_layers=wl.n_layers, n_kv_heads=wl.n_kv_heads,
                        head_dim=wl.head_dim, sections=list(wl.sections), batch=wl.n_seqs,
                        tokens=batch.total_k, revisits=R, cache=f"{wl.cache}/{wl.block_size}",
                        L=wl.L, bytes_per_step=nbytes,
                        l2=flush.describe(nbytes)),
            pct_of_hbm_measured=100.0 * value / peak, pct_of_hbm_spec_8tbs=100.0 * value / SPEC_HBM_GBS,
            us_per_revisit=1e3 * ms_per_step / R,
            token_layers_per_s=batch.total_k * wl.n_layers * world * K / total_s,
            plan_us_avg=1e3 * statistics.mean(plan_ms) if plan_ms else None,
            timing="cuda graph, %d steps per replay" % args.graph_inner if args.graph
            else "stream launches of prcr_rebind_inject, events around each step; the "
                 "roofline kernel timed over %d further steps through prcr_plan + "
                 "prcr_rebind_apply" % (min(K, 20) if split else 0),
            roofline=roof, cpu_baseline=cpu, selection_manifest=manifest,
            paper_shape=shapes, next_rows=rows,
            e2e=dict(value=e2e_value, unit=UNIT, h2d_bytes_per_step=rv.h2d_bytes(),
                     d2h_bytes_per_step=rv.d2h_bytes(), steps=args.e2e_steps),
            gpu_launches=per_step * K,
            kernels_per_step=launched or None,
            launches_counted_by="torch.profiler (CUPTI), one call" if launched
            else "two entry points per step, one kernel each",
            clocks=clk.summary(), parity=check)
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def next_rows(args):
    """The NEXT rows' headline numbers, measured inside the default run (one
    GPU, rank 0) by the same code as their own --path lines, whose JSON
    lines are captured rather than printed: the attention-driven selection on
    the workload's shape (one layer of the store; the selection reads one
    layer), from the raw store and from the position-bound cache, the
    small-batch first decode step (paper 8B shape: one sequence of 933 slots
    x 36 layers) and one whole revisit (select, rebind + inject, decode) of
    the paper 8B shape at K = 32 replayed as a CUDA graph."""
    import contextlib
    import io

    def run(fn, **kw):
        ns = argparse.Namespace(**vars(args))
        ns.__dict__.update(dict(no_cpu_baseline=True, seqs=0, layers=0, graph=False,
                                flush="auto", select_source="raw"))
        ns.__dict__.update(kw)
        buf = io.StringIO()
        with contextlib.redirect_stdout(buf):
            fn(ns)
        for line in buf.getvalue().splitlines():
            if line.startswith("{"):
                return json.loads(line)
        return None

    out = {}
    for src in ("raw", "cache"):
        d = run(run_select_path, path="select", layers=1, steps=200, warmup=10, select_source=src)
        out[f"select_{src}"] = dict(workload=d["config"]["workload"], ms=d["ms_per_step"],
                                    gbs=d["value"], frac=d["roofline"]["frac"],
                                    l2=d["config"]["l2"])
    d = run(run_decode_path, path="decode", workload="paper-8b-k32", seqs=1, max_len=933,
            steps=200, warmup=10)
    out["decode_1x933"] = dict(us=1e3 * d["ms_per_step"], gbs=d["value"], frac=d["roofline"]["frac"],
                               l2=d["config"].get("l2"))
    d = run(run_pipeline_path, path="pipeline", workload="paper-8b-k32", steps=200, warmup=10,
            graph=True)
    out["revisit_k32_graph"] = dict(us=1e3 * d["ms_per_step"], timing="one CUDA graph per %d steps"
                                    % args.graph_inner)
    out["measured_by"] = ("bench.py's select / decode / pipeline paths, run inside this call "
                          "(parity: tests/test_select*_gpu.py, test_decode_gpu.py, "
                          "test_pipeline_gpu.py)")
    return out


def _timed(fn, steps, warmup, local, flush):
    import torch
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    with Clocks(local) as clk:
        for e0, e1 in ev:
            flush()
            e0.record(stream)
            fn()
            e1.record(stream)
        torch.cuda.synchronize()
    ms = [e0.elapsed_time(e1) for e0, e1 in ev]
    return ms, clk.summary()


def _launch_keys(launched, expected, steps):
    """gpu_launches from the kernels the profiler saw one step launch, else
    from the entry points' own launch counts."""
    if launched:
        return dict(gpu_launches=len(launched) * steps, kernels_per_step=launched,
                    launches_counted_by="torch.profiler (CUPTI), one step")
    return dict(gpu_launches=expected * steps, kernels_per_step=None,
                launches_counted_by="entry points' launch counts")


def run_capture_path(args):
    """Prefill capture: every visual token of every sequence, all layers."""
    import torch
    _, _, local = dist_env()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    from paper_2606_26631_gb300 import _build
    if not _build.up_to_date():
        _build.build()
    import paper_2606_26631_gb300 as prcr
    from workloads import get, make_batch
    wl = get(args.workload)
    if args.seqs:
        wl = dataclasses.replace(wl, n_seqs=args.seqs)
    src = make_batch(wl, device=dev)  # its raw store stands in for the prefill projections
    B, nL, M, H, D = wl.n_seqs, wl.n_layers, wl.n_tokens, wl.n_kv_heads, wl.head_dim
    store_k = torch.empty_like(src.store_k); store_v = torch.empty_like(src.store_v)
    coords = torch.empty_like(src.coords)
    bs = 16
    nblk = (M + bs - 1) // bs
    perm = torch.randperm(B * nblk, device=dev, generator=torch.Generator(device=dev).manual_seed(2))
    bt = perm.view(B, nblk).to(torch.int32).contiguous()
    cache_k = torch.empty((nL, B * nblk, bs, H, D), dtype=torch.bfloat16, device=dev)
    cache_v = torch.empty_like(cache_k)
    cfg = prcr.rope_cfg(nL, H, D, wl.sections, wl.theta)
    sd = prcr.store_desc(store_k, store_v, coords)
    cd = prcr.cache_paged(cache_k, cache_v, bt)
    status = torch.zeros(1, dtype=torch.int32, device=dev)

    def step():
        for b in range(B):
            prcr.prefill_capture(cfg, sd, cd, b, 0, 0, 0, src.store_k[b], src.store_v[b],
                                 src.coords[b], status)

    step()
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert torch.equal(store_k.view(torch.int16), src.store_k.view(torch.int16))
    nbytes = B * M * nL * H * D * 2 * 6  # read k, v; write store k, v and cache k, v
    launched = kernel_launches(step)
    flush = L2Flush(dev, args.flush, nbytes)
    ms, clk = _timed(step, args.steps, args.warmup, local, flush)
    t = sum(ms) / 1e3
    peak, kind = measured_peaks()
    value = nbytes * args.steps / t / 1e9
    mc = min(M, 1024)
    kb = src.store_k[0, :, :mc].contiguous().view(torch.int16).cpu().numpy()  # [nL, mc, H, D]
    vb = src.store_v[0, :, :mc].contiguous().view(torch.int16).cpu().numpy()
    crd = src.coords[0, :mc].cpu().numpy()

    def oracle():
        from oracle import prcr_oracle as O
        for l in range(nL):
            O.prefill_capture(kb[l], vb[l], crd, D, wl.sections, wl.theta)

    cpu = oracle_leg(args, oracle, mc * nL * H * D * 2 * 6,
                     f"sequence 0 of '{wl.name}': its first {mc} visual tokens x {nL} layers x "
                     f"{H} KV heads, one layer per oracle call")
    print(json.dumps(dict(
        metric="prefill capture GB/s (read+write)", value=value, unit=UNIT, n_gpus=1,
        steps=args.steps, warmup=args.warmup, ms_per_step=1e3 * t / args.steps,
        higher_is_better=True, scaling="weak", vs_baseline=None, dtype="f32", io_dtype="bf16",
        data="synthetic", config=dict(workload=wl.name, batch=B, tokens_per_seq=M, n_layers=nL,
                                      cache="paged/16", bytes_per_step=nbytes,
                                      l2=flush.describe(nbytes)),
        roofline=dict(bound="hbm", achieved=value, peak=peak, unit="GB/s", frac=value / peak,
                      traffic=None, kernel="capture_kernel", peak_kind=f"{kind} copy (hbm_gbs)"),
        cpu_baseline=cpu, **_launch_keys(launched, B, args.steps), clocks=clk)), flush=True)


def run_decode_path(args):
    """First decode step over a populated paged cache of the workload's shape."""
    import torch
    _, _, local = dist_env()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    from paper_2606_26631_gb300 import _build
    if not _build.up_to_date():
        _build.build()
    import paper_2606_26631_gb300 as prcr
    from workloads import get, make_decode_inputs
    wl = get(args.workload)
    B = args.seqs or wl.n_seqs
    Hq = 4 * wl.n_kv_heads
    max_len = args.max_len
    inp = make_decode_inputs(B, wl.n_layers, wl.n_kv_heads, Hq, wl.head_dim, max_len, True,
                             device=dev, seed=1)
    cfg = prcr.rope_cfg(wl.n_layers, wl.n_kv_heads, wl.head_dim, wl.sections, wl.theta)
    cd = prcr.cache_paged(inp["cache_k"], inp["cache_v"], inp["block_table"])
    out = torch.empty(inp["q"].shape, dtype=torch.float32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    nws = prcr.decode_workspace_size(cfg, B, Hq, max_len)
    ws = torch.empty(max(nws, 16), dtype=torch.uint8, device=dev)

    def step():
        prcr.decode_attention(cfg, cd, inp["q"], inp["q_pos"], inp["seq_len"], max_len, out,
                              status, ws)

    step()
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    slots = int(inp["seq_len"].sum())
    nbytes = slots * wl.n_layers * wl.n_kv_heads * wl.head_dim * 2 * 2
    launched = kernel_launches(step)
    flush = L2Flush(dev, args.flush, nbytes)
    ms, clk = _timed(step, args.steps, args.warmup, local, flush)
    t = sum(ms) / 1e3
    peak, kind = measured_peaks()
    value = nbytes * args.steps / t / 1e9
    n0 = int(inp["seq_len"][0])
    s0 = torch.arange(n0, device=dev)
    blk = inp["block_table"][0][s0 // 16].long()
    K0 = inp["cache_k"][:, blk, s0 % 16].transpose(0, 1).contiguous().view(torch.int16).cpu().numpy()
    V0 = inp["cache_v"][:, blk, s0 % 16].transpose(0, 1).contiguous().view(torch.int16).cpu().numpy()
    q0 = inp["q"][0].contiguous().view(torch.int16).cpu().numpy()
    p0 = int(inp["q_pos"][0])

    def oracle():
        from oracle import prcr_oracle as O
        qv, Kv, Vv = O.bf16_bits_to_f64(q0), O.bf16_bits_to_f64(K0), O.bf16_bits_to_f64(V0)
        for l in range(wl.n_layers):
            O.decode_attention(qv[l], p0, Kv[:, l], Vv[:, l], wl.head_dim, wl.sections, wl.theta)

    cpu = oracle_leg(args, oracle, n0 * wl.n_layers * wl.n_kv_heads * wl.head_dim * 2 * 2,
                     f"sequence 0 of the batch ({n0} slots) x {wl.n_layers} layers x "
                     f"{wl.n_kv_heads} KV heads, {Hq} query heads, one layer per oracle call")
    print(json.dumps(dict(
        metric="decode attention GB/s (K/V read)", value=value, unit=UNIT, n_gpus=1,
        steps=args.steps, warmup=args.warmup, ms_per_step=1e3 * t / args.steps,
        higher_is_better=True, scaling="weak", vs_baseline=None, dtype="f32", io_dtype="bf16",
        data="synthetic", config=dict(workload=wl.name, batch=B, n_q_heads=Hq, max_len=max_len,
                                      slots=slots, cache="paged/16", bytes_per_step=nbytes,
                                      workspace_bytes=nws, l2=flush.describe(nbytes)),
        roofline=dict(bound="hbm", achieved=value, peak=peak, unit="GB/s", frac=value / peak,
                      traffic=None, kernel="decode_kernel (+ merge)",
                      peak_kind=f"{kind} copy (hbm_gbs)"),
        cpu_baseline=cpu, **_launch_keys(launched, 2 if nws else 1, args.steps), clocks=clk)),
        flush=True)


def run_select_path(args):
    """Attention-driven selection of K tokens per sequence at one layer."""
    import torch
    _, _, local = dist_env()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    from paper_2606_26631_gb300 import _build
    if not _build.up_to_date():
        _build.build()
    import paper_2606_26631_gb300 as prcr
    from workloads import get, make_batch
    wl = get(args.workload)
    if args.seqs:
        wl = dataclasses.replace(wl, n_seqs=args.seqs)
    if args.layers:
        wl = dataclasses.replace(wl, n_layers=args.layers)
    batch = make_batch(wl, device=dev)
    B, M, H, D = wl.n_seqs, wl.n_tokens, wl.n_kv_heads, wl.head_dim
    Hq, k, layer = 4 * H, max(1, batch.total_k // B), wl.n_layers - 1
    q = torch.randn((B, Hq, D), device=dev, generator=torch.Generator(device=dev).manual_seed(3)
                    ).to(torch.bfloat16)
    cfg = prcr.rope_cfg(wl.n_layers, H, D, wl.sections, wl.theta)
    sd = prcr.store_desc(batch.store_k, batch.store_v, batch.coords)
    idx = torch.empty(B * k, dtype=torch.int32, device=dev)
    sro = torch.empty(B + 1, dtype=torch.int32, device=dev)
    rto = torch.empty(B + 1, dtype=torch.int32, device=dev)
    ws = torch.empty(prcr.select_workspace_size(B, Hq, M), dtype=torch.uint8, device=dev)

    if args.select_source == "raw":
        def step():
            prcr.select_topk(cfg, sd, layer, q, batch.p_txt, k, idx, sro, rto, ws)
    else:
        # the image tokens' keys as a one-layer position-bound cache laid out
        # like the workload's cache (the store's keys serve as its values)
        img0 = torch.zeros(B, dtype=torch.int32, device=dev)
        cfg1 = prcr.rope_cfg(1, H, D, wl.sections, wl.theta)
        status = torch.zeros(1, dtype=torch.int32, device=dev)
        if batch.paged:
            bs = wl.block_size
            nblk = (M + bs - 1) // bs
            perm = torch.randperm(B * nblk, device=dev,
                                  generator=torch.Generator(device=dev).manual_seed(4))
            bt = perm.to(torch.int32).view(B, nblk).contiguous()
            ck = torch.empty((1, B * nblk, bs, H, D), dtype=torch.bfloat16, device=dev)
            flat = ck.view(B * nblk * bs, H, D)
            for b in range(B):
                s_ = torch.arange(M, device=dev)
                flat[bt[b][s_ // bs].long() * bs + s_ % bs] = batch.store_k[b, layer]
            cd = prcr.cache_paged(ck, ck, bt)
        else:
            ck = batch.store_k[:, layer:layer + 1].clone()
            cd = prcr.cache_contiguous(ck, ck)

        def step():
            prcr.select_topk_cached(cfg1, cd, 0, q, batch.p_txt, img0, M, k, idx, sro, rto, status,
                                    ws)

    nbytes = B * M * H * D * 2  # the layer's keys, read once
    launched = kernel_launches(step)
    flush = L2Flush(dev, args.flush, nbytes)
    ms, clk = _timed(step, args.steps, args.warmup, local, flush)
    t = sum(ms) / 1e3
    peak, kind = measured_peaks()
    value = nbytes * args.steps / t / 1e9
    kb0 = batch.store_k[0, layer].contiguous().view(torch.int16).cpu().numpy()  # [M, H, D]
    crd0 = batch.coords[0].cpu().numpy()
    q0 = q[0].contiguous().view(torch.int16).cpu().numpy()
    p0 = int(batch.p_txt[0])

    def oracle():
        from oracle import prcr_oracle as O
        qv = O.bf16_bits_to_f64(q0)
        if args.select_source == "raw":
            rel = O.ads_relevance(qv, p0, kb0, crd0, D, wl.sections, wl.theta)
        else:
            rel = O.ads_relevance_cached(qv, p0, O.bf16_bits_to_f64(kb0), D, wl.sections, wl.theta)
        O.ads_select(rel, k)

    cpu = oracle_leg(args, oracle, M * H * D * 2,
                     f"sequence 0 of '{wl.name}' ({M} tokens x {H} KV heads, {Hq} query heads, "
                     f"k = {k}), relevance and selection")
    print(json.dumps(dict(
        metric=f"selection GB/s ({args.select_source} keys read)", value=value, unit=UNIT, n_gpus=1,
        steps=args.steps, warmup=args.warmup, ms_per_step=1e3 * t / args.steps,
        us_per_sequence=1e6 * t / args.steps / B, higher_is_better=True, scaling="weak",
        vs_baseline=None, dtype="f32", io_dtype="bf16", data="synthetic",
        config=dict(workload=wl.name, batch=B, tokens_per_seq=M, n_q_heads=Hq, k=k, layer=layer,
                    source=args.select_source, bytes_per_step=nbytes, l2=flush.describe(nbytes)),
        roofline=dict(bound="hbm", achieved=value, peak=peak, unit="GB/s", frac=value / peak,
                      traffic=None, kernel="ads_*_kernel (whole selection step)",
                      peak_kind=f"{kind} copy (hbm_gbs)"),
        cpu_baseline=cpu, **_launch_keys(launched, 4, args.steps), clocks=clk)), flush=True)


def run_pipeline_path(args):
    """One revisit end to end on the device, as a decoder would run it: the
    revisited set chosen by attention at the last layer (k = the fewest tokens
    a sequence of the workload revisits), its raw rows rebound and appended to the active
    cache (whose context rows are data), and the first decode step over the
    grown cache at the next text position."""
    import torch
    _, _, local = dist_env()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    from paper_2606_26631_gb300 import _build
    if not _build.up_to_date():
        _build.build()
    import paper_2606_26631_gb300 as prcr
    from workloads import get, make_batch
    wl = get(args.workload)
    batch = make_batch(wl, device=dev, context="random")
    B, nL, M, H, D = wl.n_seqs, wl.n_layers, wl.n_tokens, wl.n_kv_heads, wl.head_dim
    # k: the fewest tokens any sequence of the workload revisits, so that the
    # appended span stays inside the cache rows the workload provides
    sro_h, rto_h = batch.seq_rev_off.cpu().numpy(), batch.rev_tok_off.cpu().numpy()
    Hq, k = 4 * H, max(1, int(min(rto_h[sro_h[b + 1]] - rto_h[sro_h[b]] for b in range(B))))
    gen = torch.Generator(device=dev).manual_seed(5)
    q_sel = torch.randn((B, Hq, D), device=dev, generator=gen).to(torch.bfloat16)
    q_dec = torch.randn((B, nL, Hq, D), device=dev, generator=gen).to(torch.bfloat16)
    cfg = prcr.rope_cfg(nL, H, D, wl.sections, wl.theta)
    sd = prcr.store_desc(batch.store_k, batch.store_v, batch.coords)
    idx = torch.empty(B * k, dtype=torch.int32, device=dev)
    sro = torch.empty(B + 1, dtype=torch.int32, device=dev)
    rto = torch.empty(B + 1, dtype=torch.int32, device=dev)
    ws_sel = torch.empty(prcr.select_workspace_size(B, Hq, M), dtype=torch.uint8, device=dev)
    rv = prcr.Revisit(cfg, batch.store_k, batch.store_v, batch.coords, batch.cache_k, batch.cache_v,
                      batch.block_table, sro, rto, idx, batch.p_txt, batch.cache_len_in)
    max_len = int(batch.cache_len_in.max().item()) + k
    out = torch.empty(q_dec.shape, dtype=torch.float32, device=dev)
    dstat = torch.zeros(1, dtype=torch.int32, device=dev)
    nws = prcr.decode_workspace_size(cfg, B, Hq, max_len)
    ws_dec = torch.empty(max(nws, 16), dtype=torch.uint8, device=dev)

    if args.select_source == "raw":
        def select():
            prcr.select_topk(cfg, sd, nL - 1, q_sel, batch.p_txt, k, idx, sro, rto, ws_sel)
    else:
        # ranked from the cache: the image's position-bound rows taken to be
        # the first M context slots (their values are the context data)
        if int(batch.cache_len_in.min().item()) < M:
            raise SystemExit("--select-source cache needs at least n_tokens context slots")
        img0 = torch.zeros(B, dtype=torch.int32, device=dev)
        sstat = torch.zeros(1, dtype=torch.int32, device=dev)

        def select():
            prcr.select_topk_cached(cfg, rv.cache, nL - 1, q_sel, batch.p_txt, img0, M, k, idx, sro,
                                    rto, sstat, ws_sel)

    def decode():
        prcr.decode_attention(cfg, rv.cache, q_dec, rv.next_pos, rv.cache_len_out, max_len, out,
                              dstat, ws_dec)

    def step():
        select()
        rv.run()
        decode()

    step()
    torch.cuda.synchronize()
    if rv.status_value() != 0 or int(dstat.item()) != 0:
        raise RuntimeError(f"device status {rv.status_value():#x} / {int(dstat.item()):#x}")
    launched = kernel_launches(step)
    nbytes = batch.algorithmic_bytes()
    flush = L2Flush(dev, args.flush, nbytes)
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if args.graph:
        # the three stages as one CUDA graph (no launch gaps), one replay per step
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            step()
        stream.wait_stream(side)
        torch.cuda.synchronize()
        with torch.cuda.graph(g):
            step()
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
        with Clocks(local) as clk:
            for e in ev:
                flush()
                e[0].record(stream)
                g.replay()
                e[1].record(stream)
            torch.cuda.synchronize()
        total = [e[0].elapsed_time(e[1]) * 1e3 for e in ev]
        part = [[float("nan")] for _ in range(3)]
    else:
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
        with Clocks(local) as clk:
            for e in ev:
                flush()
                e[0].record(stream)
                select()
                e[1].record(stream)
                rv.run()
                e[2].record(stream)
                decode()
                e[3].record(stream)
            torch.cuda.synchronize()
        part = [[e[i].elapsed_time(e[i + 1]) * 1e3 for e in ev] for i in range(3)]
        total = [e[0].elapsed_time(e[3]) * 1e3 for e in ev]
    print(json.dumps(dict(
        metric="revisit pipeline us per step (select + rebind/inject + first decode)",
        value=statistics.mean(total), unit="us", n_gpus=1, steps=args.steps, warmup=args.warmup,
        ms_per_step=statistics.mean(total) / 1e3, higher_is_better=False, scaling="weak",
        vs_baseline=None, dtype="f32", io_dtype="bf16", data="synthetic",
        config=dict(workload=wl.name, batch=B, tokens_per_seq=M, k=k, n_q_heads=Hq, n_layers=nL,
                    select_source=args.select_source,
                    context_slots=int(batch.cache_len_in.max().item()), rebind_bytes=nbytes,
                    l2=flush.describe(nbytes)),
        timing="one CUDA graph per step (stages not timed separately)" if args.graph
        else "stream launches, events around each stage",
        us_select=statistics.mean(part[0]), us_rebind_inject=statistics.mean(part[1]),
        us_decode=statistics.mean(part[2]), us_per_revisit=statistics.mean(total) / B,
        **_launch_keys(launched, 7, args.steps), clocks=clk.summary())), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    elif args.path == "capture":
        run_capture_path(args)
    elif args.path == "decode":
        run_decode_path(args)
    elif args.path == "select":
        run_select_path(args)
    elif args.path == "pipeline":
        run_pipeline_path(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
