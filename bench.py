"""Decode benchmark of the ResKV library on synthetic long-context workloads.

One step = one shared-softmax decode (Alg. 2) of every (layer, batch, KV head)
unit of the workload for one fresh decode query per query head, through the
C ABI as a decoder issues it: one reskv_decode_attn call per layer (layer 0 ..
L-1), the L launches captured in one CUDA graph.  Also reported: all layers
in one launch (a ceiling: it needs every layer's query up front),
end to end with host buffers, and a second workload measured the same way.
The compressed cache is built first by reskv_build_cache (Alg. 1, timed on
its own).  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   (the fp64 CPU oracle on host cores)

Under torchrun (N > 1) every rank runs an independent replica on its own GPU
(the path has no exchange step); rank 0 prints the aggregate.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2607_29591_gb300 import workloads as wl  # noqa: E402

METRIC = "compressed-decode attn tokens/s and achieved HBM GB/s (% of peak), 1 GB300"
DEFAULT_WORKLOAD = "llama8b_32l_32k_b8"
SLOT_BYTES = 2 * 128 * 2            # one K row + one V row, bf16
CSRC = os.path.join(ROOT, "paper_2607_29591_gb300", "csrc")
# ncu summaries of the two tensor-core decode kernels on the default workload,
# and the sources each summary's counters were taken from
PROFILE = os.path.join(ROOT, "profiles", "decode_kernel_llama8b_32l_32k_b8.md")
KERNEL_SOURCES = [os.path.join(CSRC, f) for f in ("decode_mma.cu", "mma_tile.cuh", "device_utils.cuh")]
PROFILE_LAYER = os.path.join(ROOT, "profiles", "decode_cluster_llama8b_32l_32k_b8_per_layer.md")
KERNEL_SOURCES_LAYER = [os.path.join(CSRC, f)
                        for f in ("decode_cluster.cu", "mma_tile.cuh", "device_utils.cuh")]


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["reskv", "reference"], default="reskv")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(wl.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--second-workload", default="long_128k_b4",
                    choices=["none"] + sorted(wl.WORKLOADS),
                    help="a second workload measured the same way (no e2e leg), reported "
                         "under second_workload")
    ap.add_argument("--comparison", default="lse", choices=["lse", "none"],
                    help="also time the paper's decode structure (main pass, residual pass, "
                         "log-sum-exp merge) on the main workload, reported under comparison")
    ap.add_argument("--decode-kernel", choices=["auto", "mma", "cluster", "fma", "lse"],
                    default="auto",
                    help="automatic plan (default: cluster kernel for launches whose units "
                         "fit on the device at once, else tensor-core stream-K), one kernel, "
                         "or the paper-style comparison path (lse: main and residual passes "
                         "merged through log-sum-exp statistics)")
    ap.add_argument("--layers", type=int, default=0,
                    help="use only this many layers (smaller profiling case)")
    ap.add_argument("--budget-mode", choices=["uniform", "adakv"], default="uniform",
                    help="uniform: every (layer, batch, KV head) keeps the budget; adakv: "
                         "construction splits each (layer, batch element)'s budget between its "
                         "KV heads with AdaKV's rule (ragged layout)")
    return ap.parse_args()


# ---------------------------------------------------------------------------
# distributed plumbing (replicas only)
# ---------------------------------------------------------------------------

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def reduce_max(x: float, world: int, device) -> float:
    """Max over ranks of a per-rank time (the job's time is the slowest rank)."""
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(per_rank_units: float, max_seconds: float, world: int) -> float:
    """Whole-job throughput: units of every rank over the slowest rank's time."""
    return per_rank_units * world / max_seconds


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.3)
        except FileNotFoundError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# roofline bookkeeping
# ---------------------------------------------------------------------------

def measured_peak_gbs():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def kernel_hash(sources=None):
    h = hashlib.sha256()
    for p in sources or KERNEL_SOURCES:
        with open(p, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(units_per_launch: int, profile=None, sources=None):
    """DRAM bytes per launch from a committed ncu summary, if the kernel
    source has not changed since it was captured (else None)."""
    profile = profile or PROFILE
    if not os.path.exists(profile):
        return None
    text = open(profile).read()
    m_hash = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]+)", text)
    m_bpu = re.search(r"dram_bytes_per_unit:\s*([0-9.]+)", text)
    if not m_hash or not m_bpu or m_hash.group(1) != kernel_hash(sources):
        return None
    return int(float(m_bpu.group(1)) * units_per_launch)


def algorithmic_bytes(n_main: np.ndarray, n_res: np.ndarray) -> int:
    """Bytes the method must read per decode step: every main and residual
    K/V row (512 B) plus the residual log-counts (4 B)."""
    return int((n_main.astype(np.int64) + n_res).sum()) * SLOT_BYTES + int(n_res.sum()) * 4


# ---------------------------------------------------------------------------
# CPU baseline: the fp64 oracle on host cores
# ---------------------------------------------------------------------------

def oracle_unit(w: wl.Workload, u: int):
    """One unit shaped like the workload's compressed cache, for timing the
    oracle: rows from the seeded generator, r from the candidate grid (or the
    workload's drawn r), seeded by the unit index."""
    import oracle as orc
    rng = np.random.default_rng([42, int(u)])
    grid = [0] + orc.candidate_budgets(w.budget, (0.05, 0.10, 0.15, 0.20))
    ws = wl.scaled(w, seq_len=max(w.budget, 64))
    l, rem = divmod(int(u), w.batch * w.n_kv_heads)
    b, h = divmod(rem, w.n_kv_heads)
    K, V = wl.unit_kv(ws, l, b, h, "cpu")
    r = int(rng.choice(grid)) if w.residual != "drawn" else int(w.residual_override()[u])
    m = w.budget - r
    Kf, Vf = K.double().numpy(), V.double().numpy()
    cnt = rng.integers(1, 300, r)
    return (orc.UnitCache(main_pos=np.arange(m), kmain=Kf[:m], vmain=Vf[:m], kbar=Kf[m:m + r],
                          vbar=Vf[m:m + r], counts=cnt, logc=np.log(cnt.astype(np.float64)), r=r),
            wl.unit_decode_queries(ws, l, b, h, K, 1)[:, 0].double().numpy())


def oracle_sample(w: wl.Workload, n: int):
    return sorted(int(u) for u in np.random.default_rng(42).choice(w.n_units, size=min(n, w.n_units),
                                                                    replace=False))


_WORKER_UNITS = {}


def _oracle_init(w, idx):
    """Process-pool initializer: every worker generates the whole sample once."""
    torch.set_num_threads(1)
    for u in idx:
        _WORKER_UNITS[u] = oracle_unit(w, u)


def _oracle_decode(args):
    """Decode the given sample units `reps` times (fp64 oracle, one process)."""
    import oracle as orc
    idx, reps = args
    cfg = orc.OracleConfig(budget=1)
    for _ in range(reps):
        for u in idx:
            un, q = _WORKER_UNITS[u]
            orc.decode_unit(un, q, cfg)
    return len(idx) * reps


class OraclePool:
    """The fp64 oracle decode on the host cores: one spawned process per core,
    each holding its part of the seeded sample.  Both CPU legs (the GPU arm's
    cpu_baseline and the reference arm) time it the same way: one dispatch =
    every worker decodes its units `reps` times, wall clock around the
    dispatch, with reps chosen so that a dispatch takes about a second and its
    inter-process cost (measured alone: a dispatch with reps = 0) is small."""

    def __init__(self, w: wl.Workload, n_sample: int, procs: int):
        import concurrent.futures
        import multiprocessing
        self.idx = oracle_sample(w, n_sample)
        self.procs = max(1, min(procs, len(self.idx)))
        self.chunks = [c.tolist() for c in np.array_split(np.array(self.idx), self.procs) if len(c)]
        self.ex = concurrent.futures.ProcessPoolExecutor(
            self.procs, mp_context=multiprocessing.get_context("spawn"),
            initializer=_oracle_init, initargs=(w, self.idx))
        self.run(1)                                  # every worker up and warm
        _, self.dispatch_s = self.run(0)
        _, t1 = self.run(1)
        self.reps = max(1, int(round(1.0 / max(t1, 1e-3))))

    def run(self, reps: int) -> tuple:
        """(unit decodes, wall seconds) of one dispatch of `reps` passes."""
        t0 = time.perf_counter()
        n = sum(self.ex.map(_oracle_decode, [(c, reps) for c in self.chunks]))
        return n, time.perf_counter() - t0

    def describe(self) -> str:
        return (f"fp64 oracle decode of {len(self.idx)} seeded units split over {self.procs} "
                f"spawned processes; one dispatch = {self.reps} passes over the sample "
                f"(inter-process cost of a dispatch alone {self.dispatch_s * 1e3:.1f} ms), "
                f"wall clock, extrapolated to all units of one step")

    def close(self):
        self.ex.shutdown()


def construction_flops(w: wl.Workload) -> dict:
    """Algorithmic flops of the dense construction stages (multiply-add = 2):
    scores 2 n_fit G s d per unit, validation targets 4 n_val G s d, Lloyd
    distances 2 T |E_r| r d per candidate r (T = 4 rounds, |E_r| = s - b + r)."""
    d, s, b, G, U, T = w.head_dim, w.seq_len, w.budget, w.group, w.n_units, 4
    out = {}
    if b >= s:
        return out
    if w.score_mode == 0:
        out["scores"] = 2 * w.n_fit * G * s * d * U
    if w.residual == "proxy":
        out["validation_targets"] = 4 * w.n_val * G * s * d * U
        rs = sorted({int(np.floor(float(np.float32(x)) * b)) for x in (0.05, 0.10, 0.15, 0.20)})
        rs = [r for r in rs if r > 0 and b - r >= w.recent_window]
        out["lloyd"] = sum(2 * T * (s - b + r) * r * d for r in rs) * U
    else:
        out["lloyd"] = sum(2 * T * (s - b + int(r)) * int(r) * d for r in w.residual_override())
    return out


def cpu_construction(w: wl.Workload, budget_s: float = 10.0):
    """The oracle's Alg. 1 on seeded units of the workload at full size, until
    about budget_s of work; per-unit time and extrapolations."""
    import oracle as orc
    f64 = lambda t: t.float().double().numpy()
    ovr = w.residual_override()
    order = np.random.default_rng(42).permutation(w.n_units)
    times = []
    t_start = time.perf_counter()
    for u in order:
        l, rem = divmod(int(u), w.batch * w.n_kv_heads)
        b, h = divmod(rem, w.n_kv_heads)
        K, V = wl.unit_kv(w, l, b, h)
        Qo = wl.unit_obs_queries(w, l, b, h, K) if w.n_obs > 0 else None
        cfg = orc.OracleConfig(budget=w.budget, recent_window=w.recent_window, n_fit=w.n_fit,
                               n_val=w.n_val, score_mode=w.score_mode,
                               residual_override=None if ovr is None else int(ovr[u]))
        t0 = time.perf_counter()
        orc.build_unit(f64(K), f64(V), None if Qo is None else f64(Qo), cfg)
        times.append(time.perf_counter() - t0)
        if time.perf_counter() - t_start > budget_s:
            break
    per_unit = float(np.mean(times))
    cores = os.cpu_count() or 1
    return {"per_unit_s": per_unit, "units_sampled": len(times),
            "extrapolated_s_one_process": per_unit * w.n_units,
            "extrapolated_s_all_cores": per_unit * w.n_units / cores,
            "how": f"fp64 oracle Alg. 1 (scores, ranking, validation proxy, Lloyd, entries) on "
                   f"{len(times)} seeded unit(s) at full size, one process each; the all-cores "
                   f"figure assumes the {w.n_units} independent units spread over {cores} cores"}


def cpu_baseline(w: wl.Workload, dispatches: int = 8):
    """The oracle as it stands on the host cores (same method as the
    reference arm), a single-thread figure, and the oracle's construction."""
    cores = os.cpu_count() or 1
    pool = OraclePool(w, 64, cores)
    n, t = 0, 0.0
    for _ in range(dispatches):
        dn, dt = pool.run(pool.reps)
        n += dn
        t += dt
    pool.close()
    step_s = t * w.n_units / n
    # one thread: the same units in this process
    import oracle as orc
    one = [oracle_unit(w, u) for u in pool.idx[:16]]
    cfg = orc.OracleConfig(budget=1)
    t0 = time.perf_counter()
    for un, q in one:
        orc.decode_unit(un, q, cfg)
    step_s1 = (time.perf_counter() - t0) * w.n_units / len(one)
    return {"value": w.batch / step_s, "unit": "tokens/s", "cores": pool.procs, "kind": "oracle",
            "sample": pool.describe() + f"; {dispatches} dispatches",
            "single_thread_value": w.batch / step_s1,
            "single_thread_sample": f"{len(one)} of those units in one process, one thread",
            "construction": cpu_construction(w)}


def run_reference(args, world, rank):
    """The reference arm: the fp64 oracle, as it stands, on the host cores;
    every step is one dispatch (cpu_baseline's method)."""
    if rank != 0:
        return
    world = 1 if world < 1 else world
    w = wl.WORKLOADS[args.workload]
    cores = os.cpu_count() or 1
    pool = OraclePool(w, 64, cores)
    for _ in range(args.warmup):
        pool.run(pool.reps)
    n_tot, t = 0, 0.0
    for _ in range(args.steps):
        n, dt = pool.run(pool.reps)
        n_tot += n
        t += dt
    pool.close()
    step_s = (t / n_tot) * w.n_units
    value = w.batch / step_s
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w, args.budget_mode, world),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": pool.procs,
                             "kind": "oracle",
                             "sample": pool.describe() + "; one dispatch per step"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def workload_config(w: wl.Workload, budget_mode: str = "uniform", world: int = 1) -> dict:
    """The JSON line's config, the same in both arms: the workload's shape,
    its budget mode, the parallelism, and why no L2 flush is needed."""
    slots = w.n_units * min(w.budget, w.seq_len) * SLOT_BYTES
    return {"workload": w.name, "layers": w.n_layers, "batch": w.batch,
            "kv_heads": w.n_kv_heads, "q_heads": w.n_q_heads, "head_dim": w.head_dim,
            "seq_len": w.seq_len, "budget": w.budget, "residual": w.residual,
            "budget_mode": budget_mode,
            "parallelism": "replicas" if world > 1 else "single GPU",
            "l2": f"inputs larger than L2: {slots / 1e9:.2f} GB of K/V slots read per step"}


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------

def build_workload(w: wl.Workload, n_q: int, device, decode_kernel: int, budget_mode: int = 0):
    """Generate inputs layer by layer; build the compressed cache (timed)."""
    from paper_2607_29591_gb300 import reskv as R
    Ks, Vs, Qs = [], [], []
    Qdec = torch.empty((n_q, w.n_layers, w.batch, w.n_q_heads, w.head_dim),
                       dtype=torch.bfloat16, device=device)
    for l in range(w.n_layers):
        K, V, Qo, Qd = wl.layer_inputs(w, l, device, n_dec_steps=n_q)
        Ks.append(K)
        Vs.append(V)
        Qs.append(Qo)
        Qdec[:, l] = Qd
    cfg = R.reskv_config_default(batch=w.batch, n_layers=w.n_layers, n_kv_heads=w.n_kv_heads,
                                 group=w.group, seq_len=w.seq_len, budget=w.budget,
                                 recent_window=w.recent_window, n_obs=w.n_obs, n_fit=w.n_fit,
                                 n_val=w.n_val, score_mode=w.score_mode,
                                 residual_override=w.residual_override(),
                                 decode_kernel=decode_kernel, budget_mode=budget_mode)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    cache = R.reskv_build_cache(cfg, Ks, Vs, Qs if w.n_obs > 0 else None)
    e1.record()
    torch.cuda.synchronize()
    build_s = e0.elapsed_time(e1) / 1e3
    R.reskv_check_status(cache)
    del Ks, Vs, Qs
    torch.cuda.empty_cache()
    return cache, Qdec, build_s


def roofline(alg_bytes: int, launch_s: float, peak: float, peak_kind: str, kernel: str,
             traffic) -> dict:
    achieved = alg_bytes / launch_s / 1e9
    return {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
            "frac": achieved / peak, "traffic": traffic, "kernel": kernel,
            "peak_kind": f"{peak_kind} (burst copy)", "algorithmic_bytes_per_launch": alg_bytes,
            "launch_us": launch_s * 1e6}


def time_per_layer(R, cache, w, Qdec, O, warmup: int, steps: int, device,
                   clk=None, world: int = 1):
    """Seconds of `steps` decode steps of one-layer calls: the L launches of a
    step (layer 0 .. L-1, reskv_decode_attn) captured in one CUDA graph; every
    step copies its fresh queries into the graph's query buffer, then replays
    it.  CUDA events on the launching stream."""
    s = torch.cuda.Stream(device)
    s.wait_stream(torch.cuda.current_stream(device))
    Qs = torch.empty_like(Qdec[0])                    # [L, B, H_q, d]

    def launches():
        for l in range(w.n_layers):
            R.reskv_decode_attn(cache, l, Qs[l], O[l], stream=s)

    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(s):
        Qs.copy_(Qdec[0])
        launches()                                    # warm, outside capture
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=s):
            launches()
        for i in range(warmup):
            Qs.copy_(Qdec[i % Qdec.shape[0]])
            graph.replay()
        s.synchronize()
        with clk if clk is not None else _nullctx():
            barrier(world)
            torch.cuda.synchronize()
            e0.record(s)
            for i in range(steps):
                Qs.copy_(Qdec[(warmup + i) % Qdec.shape[0]])
                graph.replay()
            e1.record(s)
            torch.cuda.synchronize()
            barrier(world)
    del graph
    return e0.elapsed_time(e1) / 1e3


class _nullctx:
    def __enter__(self):
        return self

    def __exit__(self, *exc):
        return False


def time_all_layer(R, cache, w, Qdec, O, warmup: int, steps: int):
    """Seconds of `steps` steps of one reskv_decode_attn(layer = -1) launch
    each (every layer in one launch), fresh queries per step."""
    stream = torch.cuda.current_stream()
    for i in range(warmup):
        R.reskv_decode_attn(cache, -1, Qdec[i % Qdec.shape[0]], O)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(steps):
        R.reskv_decode_attn(cache, -1, Qdec[(warmup + i) % Qdec.shape[0]], O)
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / 1e3


def time_e2e(R, cache, Qdec, O, warmup: int, steps: int, world: int, device) -> tuple:
    """reskv_decode_attn_host on page-locked host Q and O: the one decode
    launch reads each unit's queries from host memory and writes its outputs
    there (over the host link, overlapped with streaming the cache); the host
    waits for every step."""
    Qh = Qdec[:min(Qdec.shape[0], 64)].cpu().pin_memory()
    Oh = torch.empty(O.shape, dtype=torch.float32).pin_memory()
    stream = torch.cuda.current_stream()
    for i in range(max(3, warmup)):
        R.reskv_decode_attn_host(cache, Qh[i % Qh.shape[0]], Oh, stream=stream)
        stream.synchronize()
    barrier(world)
    t0 = time.perf_counter()
    for i in range(steps):
        R.reskv_decode_attn_host(cache, Qh[i % Qh.shape[0]], Oh, stream=stream)
        stream.synchronize()
    te = reduce_max(time.perf_counter() - t0, world, device)
    return te, int(Qh[0].numel() * 2), int(Oh.numel() * 4)


def measure(args, w: wl.Workload, R, kern: int, bmode: int, device, world: int, peak: float,
            peak_kind: str, clk=None, with_e2e: bool = True) -> dict:
    """Build the workload's cache, then time its decode step: one-layer calls
    in a CUDA graph, one
    all-layer launch, and end to end with host buffers."""
    n_q = args.steps + args.warmup
    cache, Qdec, build_s = build_workload(w, n_q, device, kern, bmode)
    info = R.reskv_get_info(cache)
    unit_budgets = R.reskv_get_unit_budgets(cache)

    def plan_name(cs, wpc):
        if kern == R.RESKV_DECODE_LSE_MERGE:
            return "paper-style: main pass + residual pass + log-sum-exp merge (3 launches)"
        if cs == 0:
            return "fma" if kern == R.RESKV_DECODE_FMA else "tensor-core stream-K"
        return f"tensor-core cluster: {cs} CTA(s) x {wpc} warps per unit"

    plan = {"all_layer": plan_name(info["all_cluster"], info["all_cluster_warps"]),
            "per_layer": plan_name(info["layer_cluster"], info["layer_cluster_warps"])}
    meta = R.reskv_export_cache(cache)
    alg = algorithmic_bytes(meta["n_main"], meta["n_res"])
    r_counts = meta["n_res"]
    del meta
    O = torch.empty((w.n_layers, w.batch, w.n_q_heads, w.head_dim), dtype=torch.float32,
                    device=device)
    L = w.n_layers
    alg_layer = alg // L
    launches_per_step = 3 * L if kern == R.RESKV_DECODE_LSE_MERGE else L
    units_layer = w.batch * w.n_kv_heads
    traffic_layer = None
    if info["layer_cluster"] > 0 and not info["ragged"] and w.name == DEFAULT_WORKLOAD:
        traffic_layer = profiled_traffic(units_layer, PROFILE_LAYER, KERNEL_SOURCES_LAYER)

    # ---- the step: one-layer calls ----
    t_local = time_per_layer(R, cache, w, Qdec, O, args.warmup, args.steps, device, clk, world)
    t = reduce_max(t_local, world, device)
    R.reskv_check_status(cache)
    per_layer = {"s": t, "us_per_step": t / args.steps * 1e6,
                 "us_per_layer_step": t / args.steps / L * 1e6,
                 "tokens_per_s": aggregate(w.batch * args.steps, t, world),
                 "roofline": roofline(alg_layer, t_local / args.steps / L, peak, peak_kind,
                                      plan["per_layer"], traffic_layer),
                 "how": f"{L} one-layer reskv_decode_attn launches per step replayed as one CUDA "
                        f"graph; each step copies fresh queries into the graph's buffer"}
    # ---- every layer in one launch ----
    t_all = time_all_layer(R, cache, w, Qdec, O, args.warmup, args.steps)
    R.reskv_check_status(cache)
    all_layer = {"us_per_step": t_all / args.steps * 1e6,
                 "us_per_layer_step": t_all / args.steps / L * 1e6,
                 "tokens_per_s": w.batch * args.steps / t_all,
                 "roofline": roofline(alg, t_all / args.steps, peak, peak_kind, plan["all_layer"],
                                      None if info["ragged"] or w.name != DEFAULT_WORKLOAD
                                      else profiled_traffic(w.n_units)),
                 "q_o_bytes_per_step": int(w.n_units * w.group * w.head_dim * (2 + 4)),
                 "how": "one reskv_decode_attn(layer=-1) launch per step (needs every layer's "
                        "query up front: a ceiling, not a decoder's step)"}
    out = {"config": workload_config(w, args.budget_mode, world),
           "run": {"mean_r": float(np.mean(r_counts)),
                   "units_with_residual": float(np.mean(r_counts > 0)),
                   "unit_budget_min_max": [int(unit_budgets.min()), int(unit_budgets.max())],
                   "decode_plan": plan,
                   "algorithmic_bytes_per_step": alg},
           "per_layer": per_layer, "all_layer": all_layer,
           "launches_per_step": launches_per_step, "construction_s": build_s,
           "construction_stages_ms": dict(zip(
               ["scores", "ranking", "validation_targets", "lloyd", "validation_loss_and_choice",
                "pack"], [round(x, 3) for x in info["build_ms"]])),
           "construction_tflops": {
               k: round(f / (info["build_ms"][i] * 1e-3) / 1e12, 2)
               for k, i in (("scores", 0), ("validation_targets", 2), ("lloyd", 3))
               for f in [construction_flops(w).get(k)] if f and info["build_ms"][i] > 0}}
    if with_e2e:
        te, bi, bo = time_e2e(R, cache, Qdec, O, args.warmup, args.steps, world, device)
        out["e2e"] = {"value": aggregate(w.batch * args.steps, te, world), "unit": "tokens/s",
                      "h2d_bytes_per_step": bi, "d2h_bytes_per_step": bo,
                      "how": "reskv_decode_attn_host on pinned host Q and O: the decode launch "
                             "reads Q from and writes O to host memory (NVLink-C2C), host waits "
                             "every step"}
    cache.free()
    del Qdec, O
    torch.cuda.empty_cache()
    return out


def main():
    args = parse_args()
    if args.impl == "reference":
        # the CPU oracle needs no process group: rank 0 runs, the others exit
        run_reference(args, int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")))
        return
    world, rank, local = dist_setup()
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    from paper_2607_29591_gb300 import build as B
    from paper_2607_29591_gb300 import reskv as R
    B.build()
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    w = wl.WORKLOADS[args.workload]
    if args.layers:
        w = wl.scaled(w, n_layers=args.layers, name=f"{w.name}_{args.layers}l")
    kern = {"auto": R.RESKV_DECODE_AUTO, "mma": R.RESKV_DECODE_MMA,
            "cluster": R.RESKV_DECODE_CLUSTER, "fma": R.RESKV_DECODE_FMA,
            "lse": R.RESKV_DECODE_LSE_MERGE}[args.decode_kernel]
    bmode = R.RESKV_BUDGET_ADAKV if args.budget_mode == "adakv" else R.RESKV_BUDGET_UNIFORM
    peak, peak_kind = measured_peak_gbs()

    # clocks are sampled around the timed region of the step
    clk = ClockSampler(local)
    main_rec = measure(args, w, R, kern, bmode, device, world, peak, peak_kind, clk=clk)
    clocks = clk.summary()
    second = None
    if args.second_workload != "none" and not args.layers:
        w2 = wl.WORKLOADS[args.second_workload]
        clk2 = ClockSampler(local)
        second = measure(args, w2, R, kern, bmode, device, world, peak, peak_kind, clk=clk2,
                         with_e2e=False)
        second["clocks"] = clk2.summary()

    comparison = None
    if args.comparison == "lse" and not args.layers and kern != R.RESKV_DECODE_LSE_MERGE:
        # the same cache built again, decoded the paper's way (3 launches per call)
        cmp = measure(args, w, R, R.RESKV_DECODE_LSE_MERGE, bmode, device, world, peak, peak_kind,
                      clk=None, with_e2e=False)
        comparison = {
            "what": "paper-style decode: main-cache pass, residual pass and a log-sum-exp merge "
                    "kernel per call (Sec. 6.1; App. B), same workload, same roofline bytes",
            "per_layer": {k: cmp["per_layer"][k] for k in ("us_per_layer_step", "tokens_per_s")},
            "per_layer_frac": cmp["per_layer"]["roofline"]["frac"],
            "all_layer": {k: cmp["all_layer"][k] for k in ("us_per_layer_step", "tokens_per_s")},
            "all_layer_frac": cmp["all_layer"]["roofline"]["frac"]}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w)

    if rank == 0:
        pl = main_rec["per_layer"]
        line = {
            "metric": METRIC, "value": pl["tokens_per_s"], "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": pl["us_per_step"] / 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": main_rec["config"],
            "run": dict(main_rec["run"], launch=f"one reskv_decode_attn(layer) launch per layer, "
                                                f"{w.n_layers} per step, in one CUDA graph"),
            "us_per_layer_step": pl["us_per_layer_step"],
            "roofline": pl["roofline"],
            "all_layer_launch": main_rec["all_layer"],
            "construction_s": main_rec["construction_s"],
            "construction_stages_ms": main_rec["construction_stages_ms"],
            "construction_tflops": main_rec["construction_tflops"],
            "e2e": main_rec["e2e"],
            "clocks": clocks,
            "gpu_launches": args.steps * main_rec["launches_per_step"],
            "cpu_baseline": cpu,
        }
        if second is not None:
            line["second_workload"] = {
                "config": second["config"], "run": second["run"], "per_layer": second["per_layer"],
                "all_layer_launch": second["all_layer"], "construction_s": second["construction_s"],
                "construction_stages_ms": second["construction_stages_ms"],
                "clocks": second["clocks"], "steps": args.steps, "warmup": args.warmup}
        if comparison is not None:
            line["comparison"] = comparison
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
