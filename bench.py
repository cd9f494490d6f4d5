#!/usr/bin/env python
"""Benchmark of the ECOKV prefill eviction pass (score -> select -> compact).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ecokv|reference] [--workload c3_b10]

A step is one call of ecokv_evict over every layer and KV head of the
workload (default: the 32768-token, 28-layer, 28/4-head Qwen2.5-VL-shaped
video prefill, bf16, W = 8, pooling 5, budget 10 % = 3277 tokens/head), with
K, V and the window queries already resident in HBM.  The inputs (1.88 GB of
K and V) are larger than the 129 MB L2, so no flush is needed between steps.

Metric: KV tokens processed per second per layer = L * H_kv * N / step time
(every cached key row of every layer is scored; H_kv * (N - B) of them are
evicted per layer).  One JSON line is printed by rank 0.

--impl reference times the fp64 CPU oracle (the only other implementation of
the method; the paper ships no code) on a bounded sample of the same workload.
Under torchrun with N > 1 every rank runs its own replica (the (layer, head)
units are independent: weak scaling, no data-path collective); the timing
uses a barrier and the maximum over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "KV tokens evicted/sec per layer at 1 GB300; % of HBM roofline (GB/s)"
UNIT = "tokens/s"
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 126 << 20       # GB300 L2
FLUSH_BYTES = 256 << 20    # written between timed steps when the inputs would fit in L2


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ecokv", "reference"], default="ecokv")
    ap.add_argument("--workload", default="c3_b10")
    ap.add_argument("--layers", type=int, default=0,
                    help="run only this many layers of the workload (small profiling captures)")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--variant", choices=["per-head", "adaptive", "vnorm", "pyramid", "centroid-nonwin", "winsor5", "mad"],
                    default="per-head",
                    help="adaptive: layer-wide budget shared by a layer's heads (ecokv_evict_adaptive); "
                         "vnorm: importance weighted by the value norms (ECOKV_FLAG_VNORM_IMP); "
                         "pyramid: PyramidKV per-layer budgets, beta 20 (ecokv_evict_layered); "
                         "centroid-nonwin: the centroid over the candidates only (ECOKV_FLAG_CENTROID_NONWIN); "
                         "winsor5: 5 %-95 % winsorised min-max of Eq. 2 (ECOKV_FLAG_WINSOR_5); "
                         "mad: MAD scaling in place of the min-max of Eq. 2 (ECOKV_FLAG_MAD)")
    ap.add_argument("--cpu-sample-units", type=int, default=0, help="0 = auto (about 10-30 s of CPU work)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="the bandwidth sweep instead of one workload: one layer, 8 KV / 32 query heads, bf16, "
                         "budget 10 %%, N = 2^10 .. 2^17, W in {1, 4, 16, 32}; one JSON line per point")
    return ap.parse_args()


# ---------------------------------------------------------------- byte model
def byte_model(w) -> dict:
    """Algorithmic bytes of one pass over the workload.

    ALG (the roofline numerator): every K row read once, the window queries
    read, the retained V rows read, the retained K and V rows written.
    BL: the same plus a full read of V (the BASELINE formula).
    """
    e = w.elem_bytes
    U = w.units
    keep = min(w.budget, w.n)
    k_bytes = U * w.n * w.d * e
    q_bytes = w.n_layers * w.h_q * w.window * w.d * e
    kept = U * keep * w.d * e
    idx_bytes = U * keep * 4
    alg = k_bytes + q_bytes + kept + 2 * kept + idx_bytes
    bl = k_bytes + k_bytes + q_bytes + 2 * kept
    return {"alg": alg, "bl": bl, "k": k_bytes, "q": q_bytes, "kept_rows": kept}


def tensor_path(w) -> bool:
    """bf16 inputs of at least 128 keys stream through the tensor-core kernel."""
    return w.dtype == "bf16" and w.n >= 128


def row_groups(w) -> int:
    """Launches of the tensor-core kernel per call: one per group of at most
    120 window rows (g * W rows per head)."""
    return (w.group * w.window + 119) // 120


def launches_per_call(w) -> int:
    """Kernels one ecokv_evict call launches: the persistent tensor-core
    streaming kernel (once per window-row group) or the two CUDA-core passes,
    then the finalize/select kernel (one thread-block cluster per head, or one
    CTA per head past 131072 candidates) and the compaction kernel."""
    return (row_groups(w) if tensor_path(w) else 2) + 2


# ---------------------------------------------------------------- ranks
def rank_workload(w, rank: int):
    """Replica of rank r: the same shapes, its own seeded inputs."""
    import dataclasses
    return dataclasses.replace(w, seed=w.seed + rank)


def max_over_ranks(x: float, world: int, device) -> float:
    """The slowest rank's value (all ranks must call this)."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world: int, units_per_rank: float, ms_step: float) -> float:
    """Whole-job throughput: every rank's units over the slowest rank's step time."""
    return world * units_per_rank / (ms_step * 1e-3)


def measured_peaks() -> tuple[float, str]:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# The sources that define the streaming kernel and the parameters it is
# launched with (item size, schedule lag, tail split): a recorded DRAM traffic
# figure is valid while these are unchanged.
STREAMING_SOURCES = ("tc_pass.cu", "tc_pass.cuh", "ptx.cuh", "finalize_select.cuh", "ecokv_internal.cuh",
                     "ecokv_api.cu")


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_06663_gb300", "csrc")
    for f in STREAMING_SOURCES:
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def traffic_record(workload: str):
    """DRAM bytes per launch of the dominant kernel from a committed ncu
    summary, valid only while the kernel sources are unchanged."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except Exception:
        return None
    r = rec.get(workload)
    if not r or r.get("source_hash") != kernel_source_hash():
        return None
    return r


# ---------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.path = None

    def start(self):
        import tempfile
        fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200",
                 "-i", str(self.dev)], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)

    def stop(self) -> dict | None:
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    rows.append((float(parts[1]), float(parts[2]), parts[4:9]))
                except ValueError:
                    continue
        os.unlink(self.path)
        if not rows:
            return None
        sm = [r[0] for r in rows]
        top = max(sm)
        loaded = [r for r in rows if r[0] >= 0.5 * top] or rows
        names = ["active", "hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in loaded:
            for n, v in zip(names[1:], r[2][1:]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(r[0] for r in loaded), "sm_max_mhz": rows[0][1],
                "reasons": sorted(reasons), "samples": len(rows)}


# ---------------------------------------------------------------- CPU oracle leg
_INPUT_CACHE: dict = {}


def _oracle_units(args):
    """Worker: run the fp64 oracle on some (layer, head) units of a workload."""
    wl_key, units = args
    import torch
    torch.set_num_threads(1)
    from oracle import ecokv_oracle as O
    from paper_2609_06663_gb300.workloads import make_inputs, workload
    w = workload(wl_key)
    n_tok = 0
    t_total = 0.0
    for (l, h) in units:
        key = (wl_key, l)
        if key not in _INPUT_CACHE:
            _INPUT_CACHE.clear()
            _INPUT_CACHE[key] = make_inputs(w, layers=range(l, l + 1))
        K, V, Q = _INPUT_CACHE[key]
        g = w.group
        Ku, Vu, Qu = K[:, h:h + 1], V[:, h:h + 1], Q[:, h * g:(h + 1) * g]
        p = O.Params(n_layers=1, h_kv=1, h_q=g, n=w.n, d=w.d, window=w.window, budget=w.budget,
                     pool_kernel=w.pool_kernel)
        t0 = time.perf_counter()
        O.evict(Ku, Vu, Qu, p)
        t_total += time.perf_counter() - t0
        n_tok += w.n
    return n_tok, t_total


def oracle_pool(cores: int):
    """A pool of spawned, single-threaded worker processes for the oracle."""
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[v] = "1"
    return mp.get_context("spawn").Pool(cores)


def cpu_oracle_rate(wl_key: str, w, n_units: int, pool, cores: int) -> dict:
    """Tokens/s of the oracle over a bounded sample of units, split across
    `cores` single-threaded workers that run in parallel."""
    units = [((i // w.h_kv) % w.n_layers, i % w.h_kv) for i in range(n_units)]
    per = [units[i::cores] for i in range(cores)]
    per = [u for u in per if u]
    t0 = time.perf_counter()
    res = pool.map(_oracle_units, [(wl_key, u) for u in per])
    wall = time.perf_counter() - t0
    n_tok = sum(r[0] for r in res)
    busy = max(r[1] for r in res)
    return {"value": n_tok / busy, "unit": UNIT, "cores": len(per), "kind": "oracle",
            "sample": f"{n_units} (layer, head) units of {w.name} ({n_tok} key rows), fp64 numpy oracle, "
                      f"{len(per)} spawned single-thread workers; rate = rows / busiest worker's compute time "
                      f"(input generation excluded); wall {wall:.1f} s"}


def default_sample_units(w, cores: int) -> int:
    # about 0.25 s of oracle time per 32k-token unit: aim for ~10-20 s of CPU work
    per_unit = 0.25 * w.n / 32768 * max(1, w.group * w.window) / 56
    return max(cores, min(4 * cores, int(15.0 / max(per_unit, 1e-3))))


# ---------------------------------------------------------------- main
def main():
    args = parse_args()
    import torch

    from paper_2609_06663_gb300.workloads import workload

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    w = workload(args.workload)
    if args.layers:
        import dataclasses
        w = dataclasses.replace(w, n_layers=args.layers, name=f"{w.name}_L{args.layers}")
    cores = max(1, min(16, os.cpu_count() or 1))

    if args.impl == "reference":
        run_reference(args, w, rank, world, cores)
        return
    if args.sweep:
        if rank == 0:
            run_sweep(args)
        return

    import torch.distributed as dist
    if world > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    from paper_2609_06663_gb300 import ecokv as E
    from paper_2609_06663_gb300.workloads import make_inputs

    K, V, Q = make_inputs(rank_workload(w, rank), device=dev)
    budgets = E.pyramid_budgets(w.n_layers, w.budget, w.window, 20.0) if args.variant == "pyramid" else None
    p = E.make_params(n_layers=w.n_layers, h_kv=w.h_kv, h_q=w.h_q, n=w.n, d=w.d, window=w.window,
                      budget=max(budgets) if budgets else w.budget, pool_kernel=w.pool_kernel,
                      flags={"vnorm": E.ECOKV_FLAG_VNORM_IMP,
                             "centroid-nonwin": E.ECOKV_FLAG_CENTROID_NONWIN,
                             "winsor5": E.ECOKV_FLAG_WINSOR_5,
                             "mad": E.ECOKV_FLAG_MAD}.get(args.variant, 0))
    ws = E.alloc_workspace(p, dev)
    n_keep = min(p.budget, w.n)
    idx = torch.empty(w.n_layers, w.h_kv, n_keep, dtype=torch.int32, device=dev)
    Ko = torch.empty(w.n_layers, w.h_kv, n_keep, w.d, dtype=K.dtype, device=dev)
    Vo = torch.empty_like(Ko)
    lam = torch.empty(w.n_layers, w.h_kv, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    dt = E.dtype_code(K)

    adaptive = args.variant == "adaptive"
    if adaptive:
        rows = w.h_kv * n_keep
        idx_a = torch.empty(w.n_layers, rows, dtype=torch.int32, device=dev)
        off_a = torch.empty(w.n_layers, w.h_kv + 1, dtype=torch.int32, device=dev)
        Ko_a = torch.empty(w.n_layers, rows, w.d, dtype=K.dtype, device=dev)
        Vo_a = torch.empty_like(Ko_a)

    lb_host = torch.tensor(budgets, dtype=torch.int32) if budgets else None

    def step():
        if adaptive:
            code = E.ecokv_evict_adaptive(p, dt, K, V, Q, idx_a, off_a, Ko_a, Vo_a, lam, ws, ws.numel(), stream)
        elif budgets:
            code = E.ecokv_evict_layered(p, dt, K, V, Q, lb_host.data_ptr(), idx, Ko, Vo, None, lam, ws, ws.numel(),
                                         stream)
        else:
            code = E.ecokv_evict(p, dt, K, V, Q, idx, Ko, Vo, None, lam, ws, ws.numel(), stream)
        if code:
            raise E.EcokvError(code, "ecokv_evict")

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    assert E.ecokv_device_status(ws, stream) == 0
    # inputs that L2 could hold between steps are flushed out of it before
    # every timed step (a 256 MB write outside the timed region)
    in_bytes = (K.numel() + V.numel() + Q.numel()) * K.element_size()
    flush_buf = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev) if in_bytes < 2 * L2_BYTES else None

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    sampler = ClockSampler(local)
    sampler.start()
    # headline: K plain steps, the library's launches back to back (each
    # kernel may be scheduled while the previous one drains)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    barrier()
    if flush_buf is None:
        ev0.record(stream)
        for i in range(args.steps):
            step()
        ev1.record(stream)
        barrier()
        ms = max_over_ranks(ev0.elapsed_time(ev1), world, dev)
    else:
        pairs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                 for _ in range(args.steps)]
        for a_, b_ in pairs:
            flush_buf.zero_()
            a_.record(stream)
            step()
            b_.record(stream)
        barrier()
        ms = max_over_ranks(sum(a_.elapsed_time(b_) for a_, b_ in pairs), world, dev)
    # per-kernel durations: K more steps with events recorded by the library
    # between its launches (streaming kernel | finalize/select | compaction)
    # on the same stream; the events order the launches strictly, so this
    # region is timed apart from the headline
    stage_ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    for evs in stage_ev:
        for e in evs:
            e.record(stream)  # creates the event handle
    barrier()
    for i in range(args.steps):
        if flush_buf is not None:
            flush_buf.zero_()
        E.ecokv_set_stage_events(stage_ev[i])
        step()
    E.ecokv_set_stage_events(None)
    barrier()
    clocks = sampler.stop()
    stage_ms = [statistics.fmean(evs[j].elapsed_time(evs[j + 1]) for evs in stage_ev) for j in range(3)]
    staged_ms_step = statistics.fmean(evs[0].elapsed_time(evs[3]) for evs in stage_ev)
    ms_step = ms / args.steps
    tokens_step = w.units * w.n
    value = job_rate(world, tokens_step, ms_step)

    # end to end through the public API for a KV cache in pinned host memory
    # (ecokv_evict_host): every call copies K and Qwin in, reads the kept V rows
    # over the host link and writes idx, K_out and V_out to host memory.
    # Consecutive calls alternate between two streams with their own
    # workspaces, so one call's copy-in overlaps the previous call's kernels.
    e2e = None
    if args.e2e_steps > 0 and args.variant == "per-head":
        hK = K.cpu().pin_memory()
        hV = V.cpu().pin_memory()
        hQ = Q.cpu().pin_memory()
        streams = [torch.cuda.Stream(dev) for _ in range(2)]
        wss = [E.alloc_workspace_host(p, dt, dev) for _ in range(2)]
        outs = [(torch.empty(idx.shape, dtype=idx.dtype).pin_memory(),
                 torch.empty(Ko.shape, dtype=Ko.dtype).pin_memory(),
                 torch.empty(Vo.shape, dtype=Vo.dtype).pin_memory()) for _ in range(2)]

        def e2e_step(i):
            s, wsh, (oi, oK, oV) = streams[i % 2], wss[i % 2], outs[i % 2]
            code = E.ecokv_evict_host(p, dt, hK, hV, hQ, oi, oK, oV, None, wsh, wsh.numel(), s)
            if code:
                raise E.EcokvError(code, "ecokv_evict_host")

        for i in range(2):
            e2e_step(i)
        barrier()
        assert torch.equal(outs[0][0], idx.cpu()) and torch.equal(outs[1][2], Vo.cpu())
        a0 = torch.cuda.Event(enable_timing=True)
        a1 = torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for s_ in streams:
            s_.wait_event(a0)
        for i in range(args.e2e_steps):
            e2e_step(i)
        for s_ in streams:
            ev = torch.cuda.Event()
            ev.record(s_)
            stream.wait_event(ev)
        a1.record(stream)
        barrier()
        e_ms = max_over_ranks(a0.elapsed_time(a1) / args.e2e_steps, world, dev)
        esz = K.element_size()
        kept_v = w.units * n_keep * w.d * esz
        e2e = {"value": job_rate(world, tokens_step, e_ms), "unit": UNIT,
               "h2d_bytes_per_step": int(hK.numel() * esz + hQ.numel() * esz + kept_v),
               "d2h_bytes_per_step": int(idx.numel() * 4 + 2 * Ko.numel() * esz),
               "ms_per_step": e_ms, "api": "ecokv_evict_host", "streams": 2,
               "h2d_detail": "K and Qwin copied in; kept V rows read by the gather from host memory"}

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    bm = byte_model(w)
    peak, peak_kind = measured_peaks()
    tr = traffic_record(args.workload)
    tc = tensor_path(w)
    # dominant kernel: the streaming pass; its algorithmic bytes are every K
    # row and the window queries read once
    stream_bytes = bm["k"] + bm["q"]
    achieved = stream_bytes / (stage_ms[0] * 1e-3) / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "traffic": tr["dram_bytes_per_launch"] if tr else None,
                "kernel": "tc_evict_kernel (streaming pass)" if tc else "score_pass1 + score_pass2 (streaming passes)",
                "alg_bytes_per_launch": stream_bytes, "launch_ms": round(stage_ms[0], 5),
                "peak_kind": f"{peak_kind} copy bandwidth (hbm_gbs)",
                "stages_ms": {"streaming": round(stage_ms[0], 5), "finalize_select": round(stage_ms[1], 5),
                              "compact": round(stage_ms[2], 5)},
                "pass": {"alg_bytes": bm["alg"], "bl_bytes": bm["bl"],
                         "alg_frac": round(bm["alg"] / (ms_step * 1e-3) / 1e9 / peak, 4),
                         "bl_frac": round(bm["bl"] / (ms_step * 1e-3) / 1e9 / peak, 4)}}

    cpu = None
    if not args.no_cpu_baseline:
        nu = args.cpu_sample_units or default_sample_units(w, cores)
        with oracle_pool(cores) as pool:
            cpu = cpu_oracle_rate(args.workload, w, nu, pool, cores)

    out = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "value_definition": "cache rows processed per second: every (layer, KV head) row of the prefill is "
                            "scored and either kept or evicted, L * H_kv * N per step; the rows evicted per "
                            "second are config.evicted_rows_per_s",
        "warmup": max(3, args.warmup), "ms_per_step": round(ms_step, 5), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if w.dtype == "bf16" else "f32",
        "data": "synthetic (seeded anisotropic + clustered/temporally correlated keys; no dataset)",
        "config": {**w.describe(), "workload": w.name,
                   "l2": "inputs larger than L2 (no flush)" if flush_buf is None else
                   "L2 flushed before every timed step (256 MB write outside the timed region)",
                   "variant": {"adaptive": "layer-wide budget (ecokv_evict_adaptive)",
                               "vnorm": "value-norm importance (ECOKV_FLAG_VNORM_IMP)",
                               "pyramid": f"per-layer budgets, PyramidKV beta 20: {budgets}",
                               "centroid-nonwin": "non-window centroid (ECOKV_FLAG_CENTROID_NONWIN)",
                               "winsor5": "5 %-95 % winsorised min-max (ECOKV_FLAG_WINSOR_5)",
                               "mad": "MAD scaling of d_E (ECOKV_FLAG_MAD)"}.get(
                                   args.variant, "per-head budget"),
                   "evicted_rows_per_s": round(job_rate(world, w.units * max(0, w.n - w.budget), ms_step), 1),
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
        # the layer-wide budget adds the layer select (3 digits x 2, count, emit) and the split
        "gpu_launches": (launches_per_call(w) + (9 if adaptive else 0) + (1 if args.variant == "vnorm" else 0)
                         # the robust forms of Eq. 2: one order-statistics launch
                         + (1 if args.variant in ("winsor5", "mad") else 0))
        * args.steps, "clocks": clocks,
        "timing": {"headline": f"{args.steps} steps back to back, CUDA events around the region",
                   "stages": f"{args.steps} further steps with per-launch events (launches serialised)",
                   "staged_ms_per_step": round(staged_ms_step, 5)},
    }
    print(json.dumps(out))
    if world > 1:
        dist.destroy_process_group()


def run_sweep(args) -> None:
    """The bandwidth sweep on GPU 0: one layer of 8 KV / 32 query heads, bf16,
    budget 10 %, N = 2^10 .. 2^17, W in {1, 4, 16, 32}.  Per point: 3 warm-up
    calls, then --steps timed calls of ecokv_evict, each after a 256 MB L2
    flush (outside the timed region), CUDA events around each call (median),
    and as many calls with the library's stage events for the per-kernel
    times.  Prints one JSON line per point."""
    import torch

    from paper_2609_06663_gb300 import ecokv as E
    from paper_2609_06663_gb300.workloads import make_inputs, sweep_workload

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    peak, peak_kind = measured_peaks()
    flush_buf = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
    steps = max(5, args.steps)
    for n in [1 << k for k in range(10, 18)]:
        for win in (1, 4, 16, 32):
            w = sweep_workload(n, win)
            K, V, Q = make_inputs(w, device=dev)
            p = E.make_params(n_layers=w.n_layers, h_kv=w.h_kv, h_q=w.h_q, n=w.n, d=w.d, window=w.window,
                              budget=w.budget, pool_kernel=w.pool_kernel)
            ws = E.alloc_workspace(p, dev)
            n_keep = min(p.budget, w.n)
            idx = torch.empty(w.n_layers, w.h_kv, n_keep, dtype=torch.int32, device=dev)
            Ko = torch.empty(w.n_layers, w.h_kv, n_keep, w.d, dtype=K.dtype, device=dev)
            Vo = torch.empty_like(Ko)
            dt = E.dtype_code(K)

            def step():
                code = E.ecokv_evict(p, dt, K, V, Q, idx, Ko, Vo, None, None, ws, ws.numel(), stream)
                if code:
                    raise E.EcokvError(code, "ecokv_evict")

            for _ in range(3):
                step()
            torch.cuda.synchronize(dev)
            assert E.ecokv_device_status(ws, stream) == 0
            pairs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                     for _ in range(steps)]
            for a_, b_ in pairs:
                flush_buf.zero_()
                a_.record(stream)
                step()
                b_.record(stream)
            stage_ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(steps)]
            for evs in stage_ev:
                for e in evs:
                    e.record(stream)
            for evs in stage_ev:
                flush_buf.zero_()
                E.ecokv_set_stage_events(evs)
                step()
            E.ecokv_set_stage_events(None)
            torch.cuda.synchronize(dev)
            ms = statistics.median(a_.elapsed_time(b_) for a_, b_ in pairs)
            stage_ms = [statistics.median(evs[j].elapsed_time(evs[j + 1]) for evs in stage_ev) for j in range(3)]
            bm = byte_model(w)
            gbs = lambda b, t: b / (t * 1e-3) / 1e9
            print(json.dumps({
                "sweep": "bandwidth sweep (one layer, 8 KV / 32 query heads, bf16, budget 10 %)",
                "workload": w.name, "n": n, "window": win, "budget": w.budget,
                "path": (f"tensor-core streaming kernel x{row_groups(w)}" if tensor_path(w) else "CUDA-core passes"),
                "ms_per_call": round(ms, 5), "tokens_per_s": round(w.units * n / (ms * 1e-3), 1),
                "evicted_rows_per_s": round(w.units * max(0, n - w.budget) / (ms * 1e-3), 1),
                "alg_gbs": round(gbs(bm["alg"], ms), 1), "bl_gbs": round(gbs(bm["bl"], ms), 1),
                "alg_frac": round(gbs(bm["alg"], ms) / peak, 4), "bl_frac": round(gbs(bm["bl"], ms) / peak, 4),
                "stages_ms": {"streaming": round(stage_ms[0], 5), "finalize_select": round(stage_ms[1], 5),
                              "compact": round(stage_ms[2], 5)},
                "streaming_frac": round(gbs(bm["k"] + bm["q"], stage_ms[0]) / peak, 4),
                "peak_gbs": peak, "peak_kind": f"{peak_kind} copy bandwidth (hbm_gbs)",
                "timing": f"median of {steps} calls, each after a 256 MB L2 flush"}), flush=True)
            del K, V, Q, ws, idx, Ko, Vo
            torch.cuda.empty_cache()


def run_reference(args, w, rank: int, world: int, cores: int) -> None:
    """The oracle timed as it stands, on host cores; rank 0 only."""
    if rank != 0:
        return
    nu = args.cpu_sample_units or max(cores, 2 * cores)
    rates = []
    with oracle_pool(cores) as pool:
        for i in range(args.warmup + args.steps):
            r = cpu_oracle_rate(args.workload, w, nu, pool, cores)
            if i >= args.warmup:
                rates.append(r)
    value = statistics.median(r["value"] for r in rates)
    cpu = dict(rates[0])
    cpu["value"] = value
    out = {"metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": round(w.units * w.n / value * 1e3, 3),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "f64", "data": "synthetic", "impl": "reference",
           "config": {**w.describe(), "workload": w.name}, "cpu_baseline": cpu,
           "timing": {"ms_per_step": "projected from the sampled rate: one step's L * H_kv * N rows divided by "
                                     f"the oracle's rows per second over {nu} sampled (layer, head) units per "
                                     "timed repetition; the whole step is not run on the CPU"},
           "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out))


if __name__ == "__main__":
    main()
