"""Benchmark of the GEM commit path on GB300.

Workload (one step = one pass of the commit path over one batch): P = 25,000,000 fp32
parameters (ResNet-50-sized), n = 100 workers, a batch of 100 commits in seeded
uniform-tick order, each with a gradient from a pool of 100 synthetic heavy-tailed
gradients (N(0, 1e-4) on 90% of coordinates, 0.01 Student-t(3) on a fixed 10%) held in
HBM.  The working set (theta, m and s of 100 workers, the pool: about 30 GB) is far larger
than L2, so no flush is needed between steps.

Metric: algorithmic HBM GB/s of the commit path, 20 bytes per parameter and commit
(g, m_w, s_w read; m_w, s_w written) plus 8 bytes per parameter and batch (theta read and
written once), and the matching commits/s.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gem|reference]
For N > 1 run under torch.distributed.run: every rank runs an independent replica on its
own GPU (no collective on the data path); the timing takes the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time
from pathlib import Path

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

METRIC = "GEM commit GB/s (% of HBM peak) at P=25M,n=100; async MLP commits/sec"
P_FULL = 25_000_000
N_WORKERS = 100
K_BATCH = 100
POOL_ROWS = 100
SEED = 5
ETA, MU, EPS = 0.01, 0.9, 1e-8
# the other commit rules (gem_mode values of include/gem.h) and kappa; bytes per parameter
# and commit moved by each rule (theta adds 8 per batch for all)
RULES = [("downpour", 1, 1.0), ("adaptive", 2, 1.0), ("kappa_sqrt_2", 3, 2.0), ("kappa_linear_2", 4, 2.0),
         ("momentum_proxy", 5, 1.0)]
RULE_BYTES = {0: 20, 1: 8, 2: 8, 3: 20, 4: 20, 5: 16}
BYTES_PER_BATCH = P_FULL * (20 * K_BATCH + 8)
FALLBACK_HBM_GBS = 6800.0

# DRAM traffic (bytes read + written) of one launch of the batched commit kernel at the
# full workload size, from an ncu capture of dram__bytes_read.sum and dram__bytes_write.sum
# on a smaller case of the same workload (P = 5,000,000, n = 100, batches of 100: about 6 GB
# on the device), scaled by P: the traffic per coordinate does not depend on P (captures at
# P = 2,500,000 and 5,000,000 agree within 1%).  Valid only for the kernel source it was
# taken on (NCU_TRAFFIC_SOURCE_SHA, a hash of the kernel's sources); null once that changes.
NCU_TRAFFIC_BYTES_PER_LAUNCH = 5 * (7_721_927_168 + 7_477_507_584) // 2   # mean of two launches at P = 5M
NCU_TRAFFIC_SOURCE_SHA = "d154547f74268928"
NCU_TRAFFIC_HOW = "two launches captured at P=5,000,000 (n=100, K=100), scaled by P to 25,000,000"


def kernel_source_sha() -> str:
    """Hash of the commit kernel's sources (the kernel and its argument block)."""
    h = hashlib.sha256()
    for name in ("gem_commit.cu", "gem_internal.h"):
        h.update((ROOT / "paper_1805_08469_gb300" / "csrc" / name).read_bytes())
    return h.hexdigest()[:16]


def measured_peaks() -> tuple[float, str]:
    f = ROOT / "MEASURED_PEAKS.json"
    try:
        d = json.loads(f.read_text())
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


class ClockSampler:
    """SM clock and throttle reasons sampled every 10 ms during the timed region.

    Reads NVML through ctypes (libnvidia-ml); nvidia-smi at 100 ms is the fallback.
    Only reads: no clock, power or mode setting is touched.
    """

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, cuda_index: int, period_s: float = 0.01):
        self.cuda_index = cuda_index
        self.period = period_s
        self.samples: list[tuple[float, float, int]] = []
        self._stop = threading.Event()
        self._thread = None
        self._proc = None
        self.source = None

    def _nvml_handle(self):
        import ctypes
        nv = ctypes.CDLL("libnvidia-ml.so.1")
        if nv.nvmlInit_v2() != 0:
            raise RuntimeError("nvmlInit failed")
        h = ctypes.c_void_p()
        bus = None
        try:
            import torch
            pr = torch.cuda.get_device_properties(self.cuda_index)
            bus = f"{pr.pci_domain_id:08x}:{pr.pci_bus_id:02x}:{pr.pci_device_id:02x}.0"
        except Exception:
            bus = None
        if bus is None or nv.nvmlDeviceGetHandleByPciBusId_v2(bus.encode(), ctypes.byref(h)) != 0:
            if nv.nvmlDeviceGetHandleByIndex_v2(self.cuda_index, ctypes.byref(h)) != 0:
                raise RuntimeError("no NVML handle")
        return nv, h

    def _run_nvml(self, nv, h):
        import ctypes
        clk = ctypes.c_uint()
        mx = ctypes.c_uint()
        rs = ctypes.c_ulonglong()
        get_reasons = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            nv.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self._stop.is_set():
            ok = nv.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0
            ok = ok and nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0
            ok = ok and get_reasons(h, ctypes.byref(rs)) == 0
            if ok:
                self.samples.append((float(clk.value), float(mx.value), int(rs.value)))
            time.sleep(self.period)

    def _run_smi(self):
        fields = ("clocks.sm,clocks.max.sm,clocks_event_reasons.hw_slowdown,"
                  "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
                  "clocks_event_reasons.sw_power_cap")
        self._proc = subprocess.Popen(["nvidia-smi", "-i", str(self.cuda_index), f"--query-gpu={fields}",
                                       "--format=csv,noheader,nounits", "-lms", "100"],
                                      stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        bits = [0x8, 0x40, 0x20, 0x4]
        for line in self._proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            try:
                r = sum(b for b, v in zip(bits, parts[2:6]) if v.lower() == "active")
                self.samples.append((float(parts[0]), float(parts[1]), r))
            except (ValueError, IndexError):
                continue

    def __enter__(self):
        try:
            nv, h = self._nvml_handle()
            self.source = "nvml"
            self._thread = threading.Thread(target=self._run_nvml, args=(nv, h), daemon=True)
        except Exception:
            self.source = "nvidia-smi"
            self._thread = threading.Thread(target=self._run_smi, daemon=True)
        self._thread.start()
        return self

    def __exit__(self, *exc):
        self._stop.set()
        if self._proc is not None:
            self._proc.terminate()
            try:
                self._proc.wait(timeout=5)
            except Exception:
                self._proc.kill()
        if self._thread is not None:
            self._thread.join(timeout=5)

    def summary(self) -> dict:
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "source": self.source}
        reasons = set()
        for _, _, r in self.samples:
            reasons.update(name for bit, name in self.REASONS.items() if r & bit)
        return {"sm_mhz": statistics.median(s[0] for s in self.samples),
                "sm_max_mhz": max(s[1] for s in self.samples), "reasons": sorted(reasons),
                "samples": len(self.samples), "source": self.source}


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
        pg = dist
    return world, rank, local, pg


def max_over_ranks(pg, value: float) -> float:
    if pg is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def barrier(pg):
    if pg is not None:
        pg.barrier()


# ------------------------------------------------------------------------- CPU oracle

ORACLE_SAMPLE = 250_000


class OracleSample:
    """The oracle's commit loop on coordinates [0, S) of the workload: inputs drawn once by
    the host generators, state carried from one timed run to the next."""

    def __init__(self, S: int, seed: int, max_batches: int = 200):
        import numpy as np

        import oracle
        from paper_1805_08469_gb300 import synth

        self.S = S
        self.order, _ = oracle.schedule_uniform(seed, N_WORKERS, max_batches * K_BATCH)
        cols = np.arange(S)
        self.theta = synth.theta0_flat(seed, cols)
        self.pool = np.stack([synth.grad_heavytail(seed, r, cols) for r in range(POOL_ROWS)])
        self.m = np.zeros((N_WORKERS, S), np.float32)
        self.s = np.tile(self.theta, (N_WORKERS, 1))
        self.next = 0
        oracle.lib()

    def run(self, batches: int) -> float:
        """Time `batches` batches of K_BATCH commits; returns seconds."""
        import numpy as np

        import oracle

        t0, t1 = self.next * K_BATCH, (self.next + batches) * K_BATCH
        if t1 > len(self.order):
            self.next, t0, t1 = 0, 0, batches * K_BATCH
        order = self.order[t0:t1]
        gidx = np.arange(t0, t1) % POOL_ROWS
        start = time.perf_counter()
        oracle.gem_run(self.theta, self.m, self.s, self.pool, order, grad_index=gidx,
                       eta=ETA, mu=MU, eps=EPS)
        dt = time.perf_counter() - start
        self.next += batches
        return dt


def oracle_mlp_rates(seconds_target: float = 4.0) -> dict:
    """The oracle's end-to-end simulation (gradients in double, OpenMP over outputs, the
    fp32 commit) on the first commits of each MLP workload, inputs from the host
    generators: commits per second on the host cores."""
    import numpy as np

    import oracle
    from paper_1805_08469_gb300 import synth

    out = {}
    for name, dims, n, b, precision, schedule, seed, _w, _t in MLP_WORKLOADS:
        P = synth.mlp_param_count(dims)
        sched = oracle.schedule_uniform if schedule == "uniform" else oracle.schedule_queue
        order = np.asarray(sched(seed, n, 400)[0], np.int32)
        batches = synth.schedule_batches(seed, order, b)
        theta = synth.xavier_theta0(seed, dims)
        m = np.zeros((n, P), np.float32)
        s_ = np.tile(theta, (n, 1))

        def run(t0, t1):
            rows, inv = np.unique(batches[t0:t1], return_inverse=True)
            X = synth.data_rows(seed, rows, dims[0])
            y = synth.teacher_labels(seed, rows, dims[0], dims[-1])
            local = inv.reshape(batches[t0:t1].shape).astype(np.int32)
            start = time.perf_counter()
            oracle.mlp_sim_run(dims, theta, m, s_, order[t0:t1], X, y, local, eta=ETA, mu=MU,
                               eps=EPS, tf32=precision == 1)
            return time.perf_counter() - start

        dt1 = run(0, 1)
        T = max(1, min(399, int(seconds_target / max(dt1, 1e-4))))
        dt = run(1, 1 + T)
        out[name] = {"commits_per_s": round(T / dt, 2), "commits": T, "seconds": round(dt, 2)}
    out["threads"] = oracle.threads()
    return out


def host_threads() -> int:
    """Host cores available to this process (the oracle's OpenMP thread count)."""
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(seconds_target: float = 12.0) -> dict:
    """The oracle's commit loop on a bounded sample of the workload, once on every host
    core (its coordinates split across threads, which changes no result) and once on one
    thread, plus the oracle's end-to-end MLP rates."""
    import oracle
    cores = host_threads()
    out = {}
    for threads in (cores, 1):
        prev = oracle.set_commit_threads(threads)
        try:
            sample = OracleSample(ORACLE_SAMPLE, SEED)
            dt1 = sample.run(1)
            batches = max(1, min(150, int(seconds_target / max(dt1, 1e-3))))
            dt = sample.run(batches)
        finally:
            oracle.set_commit_threads(prev)
        S, T = ORACLE_SAMPLE, batches * K_BATCH
        gbs = S * (20 * T + 8 * batches) / dt / 1e9
        out[threads] = {"value": round(gbs, 3), "unit": "GB/s", "cores": threads, "kind": "oracle",
                        "sample": f"coordinates [0, {S}) of P={P_FULL}, n={N_WORKERS}: {batches} batches "
                                  f"of {K_BATCH} commits in {dt:.1f} s on {threads} thread(s); same "
                                  "algorithmic bytes per coordinate",
                        "commits_per_s_scaled_to_P": round(T / dt * S / P_FULL, 3)}
    line = dict(out[cores])
    if cores != 1:
        line["single_thread"] = out[1]
    line["oracle_threads_available"] = oracle.threads()
    line["async_mlp_oracle"] = oracle_mlp_rates()
    return line


def run_reference(args, world, rank, pg):
    """Reference arm: the oracle as it stands, on the host cores, one bounded sample per step."""
    if rank != 0:
        return
    import oracle
    S = ORACLE_SAMPLE
    cores = host_threads()
    oracle.set_commit_threads(cores)
    sample = OracleSample(S, SEED, max_batches=args.warmup + args.steps + 1)
    for _ in range(args.warmup):
        sample.run(1)
    total = sum(sample.run(1) for _ in range(args.steps))
    gbs = S * (20 * K_BATCH + 8) * args.steps / total / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": round(gbs, 3), "unit": "GB/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(1e3 * total / args.steps, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "gem_commit_batch P=25M n=100, batches of 100 commits, heavy-tailed gradient pool",
                   "P": P_FULL, "n": N_WORKERS, "commits_per_step": K_BATCH,
                   "sample": f"coordinates [0, {S}) per step"},
        "cpu_baseline": {"value": round(gbs, 3), "unit": "GB/s", "cores": cores, "kind": "oracle",
                         "sample": f"coordinates [0, {S}) of P={P_FULL}, one batch of {K_BATCH} commits "
                                   f"per step, the coordinates split over {cores} thread(s)"},
        "e2e": {"value": round(gbs, 3), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------- GPU arm

def run_gem(args, world, rank, local, pg):
    import numpy as np
    import torch

    from paper_1805_08469_gb300 import gem, sim, synth_gpu

    global P_FULL, N_WORKERS, K_BATCH, POOL_ROWS, BYTES_PER_BATCH
    P_FULL, N_WORKERS, K_BATCH, POOL_ROWS = args.P, args.workers, args.batch, args.pool
    BYTES_PER_BATCH = P_FULL * (20 * K_BATCH + 8)
    torch.cuda.set_device(local)
    seed = SEED + rank
    stream = torch.cuda.Stream()
    steps_total = args.warmup + args.steps
    # the rule and factor-statistics sections reuse batches 0..10
    order, _ = sim.gem_schedule_uniform(seed, N_WORKERS, max(steps_total, 11) * K_BATCH)

    with torch.cuda.stream(stream):
        G = gem.Gem(P_FULL, N_WORKERS, ETA, MU, EPS, stream=stream)
        theta0 = synth_gpu.theta0_flat(seed, torch.empty(P_FULL, device="cuda"), stream=stream)
        G.set_theta(theta0)
        pool = torch.empty((POOL_ROWS, P_FULL), device="cuda")
        synth_gpu.grad_heavytail(seed, 0, pool, P_FULL, stream=stream)
        stream.synchronize()

        def batch(b):
            ks = range(b * K_BATCH, (b + 1) * K_BATCH)
            return [int(order[k]) for k in ks], [pool[k % POOL_ROWS] for k in ks]

        for b in range(args.warmup):
            G.commit_batch(*batch(b))
        stream.synchronize()
        barrier(pg)
        starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        launches0 = G.launches()
        batches = [batch(args.warmup + i) for i in range(args.steps)]
        with ClockSampler(local) as clocks:
            torch.cuda.synchronize()
            for i in range(args.steps):
                starts[i].record(stream)
                G.commit_batch(*batches[i])
                ends[i].record(stream)
            torch.cuda.synchronize()
        launches = G.launches() - launches0
        per_step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
        total_ms = starts[0].elapsed_time(ends[-1])
        total_ms = max_over_ranks(pg, total_ms)
        barrier(pg)
        # the fewest bytes a batch can move: every gradient read once, theta read and
        # written once, and m_w, s_w read and written once per distinct worker of the batch
        distinct = [len(set(o)) for o, _g in batches]
        reuse_min_bytes = P_FULL * (4 * K_BATCH + 8 + 16 * sum(distinct) / len(distinct))

        # single commits (one gem_commit call each, 28 bytes per parameter: g, m_w, s_w and
        # theta read, m_w, s_w and theta written) on the same state, back to back
        single = None
        if not args.no_single:
            n_single = max(20, min(4 * args.steps, 200))
            singles = [(int(order[k]), pool[k % POOL_ROWS]) for k in range(n_single)]
            for w, g in singles[:5]:
                G.commit(w, g)
            stream.synchronize()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for w, g in singles:
                G.commit(w, g)
            e1.record(stream)
            e1.synchronize()
            ms_single = e0.elapsed_time(e1) / n_single
            gbs_single = 28 * P_FULL / (ms_single * 1e-3) / 1e9
            single = {"commits_per_s": round(1e3 / ms_single, 1), "ms_per_commit": round(ms_single, 5),
                      "GB_per_s": round(gbs_single, 1), "commits": n_single,
                      "bytes_per_param": 28, "kernel": "commit_batch_kernel (one commit per launch)",
                      "note": "gem_commit calls back to back at P=25M, n=100; each launch waits on "
                              "its predecessor, so ms_per_commit bounds the kernel time from above"}

        # the other commit rules on the same workload, each with its own algorithmic bytes
        rules = None
        if not args.no_rules:
            rules = {}
            rule_steps = max(3, min(args.steps, 10))
            for name, mode, kappa in RULES:
                G.set_mode(mode, kappa)
                G.commit_batch(*batch(0))
                ms = time_batches(G, [batch(i) for i in range(rule_steps)], stream)
                bpb = P_FULL * (RULE_BYTES[mode] * K_BATCH + 8)
                rules[name] = {"GB_per_s": round(bpb / (ms * 1e-3) / 1e9, 1),
                               "commits_per_s": round(K_BATCH / (ms * 1e-3), 1),
                               "ms_per_batch": round(ms, 4),
                               "bytes_per_param_and_commit": RULE_BYTES[mode]}
            G.set_mode(gem.GEM_MODE_GEM)

        # scaling-factor statistics: every commit of a batch records its factors, then the
        # exact median of each commit's P factors
        pi_stats = None
        if not args.no_rules:
            pi_rows = torch.empty((K_BATCH, P_FULL), device="cuda")
            rows = [pi_rows[k] for k in range(K_BATCH)]
            reps = 3
            lo = torch.empty((reps + 1, K_BATCH, 1), device="cuda")
            hi = torch.empty((reps + 1, K_BATCH, 1), device="cuda")
            G.commit_batch_pi(*batch(0), rows)
            G.pi_median(rows, [0, P_FULL], lo[reps], hi[reps])
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(3 * reps)]
            stream.synchronize()
            for r in range(reps):
                ev[3 * r].record(stream)
                G.commit_batch_pi(*batch(r + 1), rows)
                ev[3 * r + 1].record(stream)
                G.pi_median(rows, [0, P_FULL], lo[r], hi[r])
                ev[3 * r + 2].record(stream)
            ev[-1].synchronize()
            commit_ms = sum(ev[3 * r].elapsed_time(ev[3 * r + 1]) for r in range(reps)) / reps
            select_ms = sum(ev[3 * r + 1].elapsed_time(ev[3 * r + 2]) for r in range(reps)) / reps
            # the same batches through the fused call: the commit kernel counts each row's
            # zeros, and rows whose medians lie in the run of zeros are not read again
            flo = torch.empty((reps, K_BATCH, 1), device="cuda")
            fhi = torch.empty((reps, K_BATCH, 1), device="cuda")
            G.commit_batch_pi_median(*batch(reps + 1), rows, [0, P_FULL], flo[0], fhi[0])
            fev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
            stream.synchronize()
            fev[0].record(stream)
            for r in range(reps):
                G.commit_batch_pi_median(*batch(reps + 2 + r), rows, [0, P_FULL], flo[r], fhi[r])
            fev[1].record(stream)
            fev[1].synchronize()
            fused_ms = fev[0].elapsed_time(fev[1]) / reps
            # bytes the selection needs: one pass of 4 bytes per factor for a row whose two
            # middle elements lie in its run of exact +0 (resolved by the first pass), three
            # passes otherwise
            lo_h = lo[:reps].cpu().numpy().reshape(reps, K_BATCH).view(np.uint32)
            hi_h = hi[:reps].cpu().numpy().reshape(reps, K_BATCH).view(np.uint32)
            one_pass = (lo_h == 0) & (hi_h == 0)
            passes = np.where(one_pass, 1, 3)
            sel_bytes = 4 * P_FULL * passes.sum() / reps
            pi_stats = {
                "commit_with_pi_ms": round(commit_ms, 4),
                "commit_with_pi_GB_per_s": round(P_FULL * (24 * K_BATCH + 8) / (commit_ms * 1e-3) / 1e9, 1),
                "median_ms": round(select_ms, 4),
                "median_Gfactors_per_s": round(K_BATCH * P_FULL / (select_ms * 1e-3) / 1e9, 2),
                "median_GB_per_s": round(sel_bytes / (select_ms * 1e-3) / 1e9, 1),
                "median_bytes": "4 per factor and pass: 1 pass for a row whose medians lie in its run "
                                "of exact +0, else 3",
                "median_rows_in_one_pass": int(one_pass.sum()),
                "median_rows": int(reps * K_BATCH),
                "commits_per_s_with_median_separate_calls": round(K_BATCH / ((commit_ms + select_ms) * 1e-3), 1),
                "fused_ms": round(fused_ms, 4),
                "commits_per_s_with_median": round(K_BATCH / (fused_ms * 1e-3), 1),
                "fused_note": "gem_commit_batch_pi_median: factors recorded and their +0 counts taken "
                              "by the commit kernel; rows whose medians lie in the run of zeros "
                              "are not read again",
                "median_pi_last_batch": float(lo[reps - 1, -1, 0]),
            }
            del pi_rows, rows

        # end to end through the public API: gradients in pinned host memory, read by the
        # commit kernel in place over the host link every step, and theta read back to the
        # host after each step
        e2e = None
        if not args.no_e2e:
            host_rows = 16
            host_pool = [pool[r].cpu().pin_memory() for r in range(host_rows)]
            theta_host = torch.empty(P_FULL, dtype=torch.float32).pin_memory()
            e2e_steps = max(2, min(args.steps, 5))

            def host_batch(b):
                ks = range(b * K_BATCH, (b + 1) * K_BATCH)
                return [int(order[k]) for k in ks], [host_pool[k % host_rows] for k in ks]

            G.commit_batch_host(*host_batch(0))
            gem.gem_read_theta(G.h, theta_host)
            G.sync()
            barrier(pg)
            t0 = time.perf_counter()
            for i in range(e2e_steps):
                G.commit_batch_host(*host_batch(i))
                gem.gem_read_theta(G.h, theta_host)
                G.sync()
            e2e_s = max_over_ranks(pg, time.perf_counter() - t0)
            e2e = {"value": round(world * BYTES_PER_BATCH * e2e_steps / e2e_s / 1e9, 1), "unit": "GB/s",
                   "h2d_bytes_per_step": K_BATCH * P_FULL * 4, "d2h_bytes_per_step": P_FULL * 4,
                   "steps": e2e_steps, "commits_per_s": round(world * K_BATCH * e2e_steps / e2e_s, 1),
                   "host_gradients": f"{host_rows} distinct pinned host buffers reused cyclically, "
                                     "read in place by the commit kernel (host link about 210 GB/s)"}
        G.close()
    del pool
    torch.cuda.empty_cache()

    flat = None if args.no_flat else run_flat_commits(seed_offset=rank)
    mlp = None if args.no_mlp else run_mlp_workloads(args, seed_offset=rank)
    cnn_out = None if args.no_mlp else run_cnn_workloads(args, seed_offset=rank)

    if rank != 0:
        return
    peak, peak_src = measured_peaks()
    avg_launch_ms = sum(per_step_ms) / len(per_step_ms)
    achieved = BYTES_PER_BATCH / (avg_launch_ms * 1e-3) / 1e9
    value = world * BYTES_PER_BATCH * args.steps / (total_ms * 1e-3) / 1e9
    traffic = NCU_TRAFFIC_BYTES_PER_LAUNCH if NCU_TRAFFIC_SOURCE_SHA == kernel_source_sha() else None
    if single is not None:
        single["frac_of_hbm_peak"] = round(single["GB_per_s"] / peak, 4)
        single["frac_of_8tbs_nominal"] = round(single["GB_per_s"] / 8000.0, 4)
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(total_ms / args.steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": f"gem_commit_batch P={P_FULL} n={N_WORKERS}, batches of {K_BATCH} commits, "
                               f"heavy-tailed gradient pool of {POOL_ROWS}",
                   "P": P_FULL, "n": N_WORKERS, "commits_per_step": K_BATCH, "pool_gradients": POOL_ROWS,
                   "eta": ETA, "mu": MU, "eps": EPS, "schedule": "uniform tick, seed 5 + rank",
                   "l2": "inputs larger than L2 (about 30 GB working set), no flush",
                   "parallelism": f"{world} independent replica(s)"},
        "commits_per_s": round(world * K_BATCH * args.steps / (total_ms * 1e-3), 1),
        "value_basis": "algorithmic bytes (20 B per parameter and commit + 8 B per parameter and "
                       "batch) over the CUDA-event launch time; a repeated worker's m_w, s_w kept "
                       "on chip count as moved, so the DRAM-based rate is roofline.dram_gbs",
        "frac_of_hbm_peak": round(value / world / peak, 4),
        "frac_of_8tbs_nominal": round(value / world / 8000.0, 4),
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": traffic,
                     "peak_source": f"{peak_src} copy bandwidth (burst)",
                     "kernel": "commit_batch_kernel", "algorithmic_bytes_per_launch": BYTES_PER_BATCH,
                     "launch_ms_min": round(min(per_step_ms), 4), "launch_ms_max": round(max(per_step_ms), 4),
                     # the DRAM rate the captured traffic implies, and the rate of the fewest
                     # bytes a batch with its repeated workers can move, both against the peak
                     "dram_gbs": None if traffic is None else
                     round(traffic / (avg_launch_ms * 1e-3) / 1e9, 1),
                     "dram_frac": None if traffic is None else
                     round(traffic / (avg_launch_ms * 1e-3) / 1e9 / peak, 4),
                     "traffic_how": NCU_TRAFFIC_HOW,
                     "reuse_min_bytes_per_launch": int(reuse_min_bytes),
                     "reuse_min_frac": round(reuse_min_bytes / (avg_launch_ms * 1e-3) / 1e9 / peak, 4),
                     "distinct_workers_per_batch": round(sum(distinct) / len(distinct), 2)},
        "single_commit": single,
        "gpu_launches": int(launches),
        "commit_rules": rules,
        "pi_statistics": pi_stats,
        "flat_single_commits": flat,
        "async_mlp": mlp,
        "async_cnn": cnn_out,
        "clocks": clocks.summary(),
        "e2e": e2e,
    }
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline()
    print(json.dumps(line), flush=True)


def time_batches(G, batches, stream) -> float:
    """Mean CUDA-event time (ms) of one gem_commit_batch call over `batches`."""
    import torch
    stream.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for order, grads in batches:
        G.commit_batch(order, grads)
    t1.record(stream)
    t1.synchronize()
    return t0.elapsed_time(t1) / len(batches)


def run_flat_commits(seed_offset: int = 0) -> dict:
    """Flat P = 1.2M, n = 20, 5,000 uniform-tick commits with log-uniform gradient scales
    (sigma_j in [1e-4, 1e-1]); the gradients cycle through a device pool of 200.  The state
    (about 0.2 GB) is L2-scale, so the GB/s are effective, not DRAM, rates."""
    import numpy as np
    import torch

    from paper_1805_08469_gb300 import gem, sim, synth, synth_gpu
    P, n, T, pool_rows, seed = 1_200_000, 20, 5000, 200, 2 + seed_offset
    stream = torch.cuda.Stream()
    order, _ = sim.gem_schedule_uniform(seed, n, T)
    out = {}
    with torch.cuda.stream(stream):
        sigma = torch.from_numpy(synth.sigma_loguniform(seed, np.arange(P))).cuda()
        pool = torch.empty((pool_rows, P), device="cuda")
        for r in range(pool_rows):
            synth_gpu.grad_loguniform(seed, r, sigma, pool[r], stream=stream)
        with gem.Gem(P, n, ETA, MU, EPS, stream=stream) as G:
            G.set_theta(synth_gpu.theta0_flat(seed, torch.empty(P, device="cuda"), stream=stream))
            grads = [pool[t % pool_rows] for t in range(T)]
            G.commit_batch([int(w) for w in order[:200]], grads[:200])      # warm-up
            ms = time_batches(G, [([int(w) for w in order], grads)], stream)
            out["batched"] = {"commits_per_s": round(T / (ms * 1e-3), 1),
                              "effective_GB_per_s": round(P * (20 * T + 8 * ((T + 199) // 200)) / (ms * 1e-3) / 1e9, 1),
                              "note": "gem_commit_batch of all 5,000 commits (launches of 200)"}
            G.sync()
            t0 = torch.cuda.Event(enable_timing=True)
            t1 = torch.cuda.Event(enable_timing=True)
            t0.record(stream)
            for t in range(T):
                G.commit(int(order[t]), grads[t])
            t1.record(stream)
            t1.synchronize()
            ms = t0.elapsed_time(t1)
            out["single"] = {"commits_per_s": round(T / (ms * 1e-3), 1),
                             "effective_GB_per_s": round(P * 28 * T / (ms * 1e-3) / 1e9, 1),
                             "note": "one gem_commit call per commit (host-issue bound)"}
    out["workload"] = f"flat P={P} n={n}, {T} uniform-tick commits, log-uniform sigma, pool of {pool_rows}"
    return out


MLP_WORKLOADS = [
    # (name, dims, n, batch, precision, schedule, seed, warmup commits, timed commits)
    ("mlp784-1000-1000-10_n100_b128_tf32", [784, 1000, 1000, 10], 100, 128, 1, "uniform", 4, 200, 2000),
    ("mlp784-1000-1000-10_n30_b128_fp32", [784, 1000, 1000, 10], 30, 128, 0, "queue", 3, 100, 1000),
    ("mlp784-64-10_n4_b32_fp32", [784, 64, 10], 4, 32, 0, "uniform", 1, 100, 1000),
]


def run_mlp_workloads(args, seed_offset: int = 0) -> dict:
    """Asynchronous GEM on the MLPs: the batched worker forward/backward over stale
    snapshots plus the in-order commits, timed with CUDA events on the handle's stream."""
    import torch

    from paper_1805_08469_gb300 import gem, sim, synth, synth_gpu

    out = {}
    stream = torch.cuda.Stream()
    X = torch.empty((synth.DATA_ROWS, 784), device="cuda")
    y = torch.empty(synth.DATA_ROWS, dtype=torch.int32, device="cuda")
    for name, dims, n, b, prec, sched, seed, warm, timed in MLP_WORKLOADS:
        if args.mlp_workload and name != args.mlp_workload:
            continue
        seed = seed + seed_offset
        if args.mlp_commits:
            warm, timed = min(warm, args.mlp_commits), args.mlp_commits
        synth_gpu.data(seed, X, y, dims[-1], stream=stream)
        pi_commits = min(timed, 500)      # then per-tensor factor medians on further commits
        T = warm + timed + pi_commits
        schedule = sim.gem_schedule_uniform if sched == "uniform" else sim.gem_schedule_queue
        order = schedule(seed, n, T)[0]
        batches = synth.schedule_batches(seed, order, b)
        P = synth.mlp_param_count(dims)
        with torch.cuda.stream(stream):
            G = gem.Gem(P, n, ETA, MU, EPS, stream=stream)
            th0 = synth_gpu.xavier(seed, dims, torch.empty(P, device="cuda"), stream=stream)
            G.set_theta(th0)
            M = sim.gem_mlp_create(G.h, dims, b, prec)
            sim.gem_mlp_set_data(M, X, y)
            losses = torch.empty(T, device="cuda")
            sim.gem_mlp_run(M, order[:warm], batches[:warm], losses[:warm])
            stream.synchronize()
            segs = len(sim.gem_plan_segments(order[warm:warm + timed], n)) - 1
            l0 = G.launches()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            sim.gem_mlp_run(M, order[warm:warm + timed], batches[warm:warm + timed],
                            losses[warm:warm + timed])
            e1.record(stream)
            stream.synchronize()
            ms = e0.elapsed_time(e1)
            commit_launches = G.launches() - l0
            lh = losses[:warm + timed].cpu().numpy()
            nt = 2 * (len(dims) - 1)
            pi_lo = torch.empty((pi_commits, nt), device="cuda")
            pi_hi = torch.empty((pi_commits, nt), device="cuda")
            a = warm + timed
            sim.gem_mlp_run_pi(M, order[a:a + 1], batches[a:a + 1], pi_lo[:1], pi_hi[:1])
            e0.record(stream)   # the first call allocated the factor rows and select scratch
            sim.gem_mlp_run_pi(M, order[a + 1:], batches[a + 1:], pi_lo[1:], pi_hi[1:], losses[a + 1:])
            e1.record(stream)
            stream.synchronize()
            ms_pi = e0.elapsed_time(e1)
            med = pi_lo.cpu().numpy()[-100:].mean(axis=0)
            sim.gem_mlp_destroy(M)
            G.close()
        gflop = 2.0 * b * sum(dims[l] * dims[l + 1] for l in range(len(dims) - 1)) * 3 - \
            2.0 * b * dims[0] * dims[1]  # forward, weight gradients, input gradients past layer 1
        out[name] = {"commits_per_s": round(timed / (ms * 1e-3), 1), "ms": round(ms, 3),
                     "commits": timed, "segments": segs, "precision": "tf32" if prec else "fp32",
                     "worker_gflop_per_commit": round(gflop / 1e9, 4),
                     "achieved_tflops": round(gflop * timed / (ms * 1e-3) / 1e12, 2),
                     "commit_launches": int(commit_launches),
                     "loss_first_100": round(float(lh[:100].mean()), 4),
                     "loss_last_100": round(float(lh[-100:].mean()), 4),
                     "with_pi_medians": {"commits_per_s": round((pi_commits - 1) / (ms_pi * 1e-3), 1),
                                         "commits": pi_commits - 1,
                                         "median_pi_per_tensor_last_100": [round(float(v), 5) for v in med]}}
    return out


CNN_WORKLOADS = [
    # (name, n, batch, seed, warmup commits, timed commits); the paper's MNIST settings
    # eta = 0.05, mu = 0.9, b = 64, uniform-tick schedule
    ("cnn_mnist_n30_b64", 30, 64, 6, 100, 1000),
    ("cnn_mnist_n100_b64", 100, 64, 7, 100, 1000),
]
CNN_ETA = 0.05


def run_cnn_workloads(args, seed_offset: int = 0) -> dict:
    """Asynchronous GEM on the MNIST convolutional network of Appendix A (synthetic 28 x 28
    images: a +-0.5 class template on 4 x 4 cells plus N(0, 1) pixel noise): commits/s
    with CUDA events, and the minibatch loss at the start and end of the timed run."""
    import torch

    from paper_1805_08469_gb300 import cnn, gem, sim, synth, synth_gpu

    out = {}
    stream = torch.cuda.Stream()
    shape = cnn.CNN_MNIST
    P = cnn.gem_cnn_param_count(shape)
    X = torch.empty((synth.DATA_ROWS, 784), device="cuda")
    y = torch.empty(synth.DATA_ROWS, dtype=torch.int32, device="cuda")
    for name, n, b, seed, warm, timed in CNN_WORKLOADS:
        seed = seed + seed_offset
        if args.mlp_commits:
            warm, timed = min(warm, args.mlp_commits), args.mlp_commits
        pi_commits = min(timed, 500)      # then per-tensor factor medians on further commits
        T = warm + timed + pi_commits
        synth_gpu.cnn_data(seed, X, y, 10, stream=stream)
        order = sim.gem_schedule_uniform(seed, n, T)[0]
        batches = synth.schedule_batches(seed, order, b)
        with torch.cuda.stream(stream):
            drop = synth_gpu.dropout(seed, 0, torch.empty((T, b, shape[2]), device="cuda"), stream=stream)
            G = gem.Gem(P, n, CNN_ETA, MU, EPS, stream=stream)
            G.set_theta(synth_gpu.cnn_theta0(seed, shape, torch.empty(P, device="cuda"), stream=stream))
            net = cnn.gem_cnn_create(G.h, shape, b)
            cnn.gem_cnn_set_data(net, X, y)
            losses = torch.empty(T, device="cuda")
            cnn.gem_cnn_run(net, order[:warm], batches[:warm], drop[:warm], losses[:warm])
            stream.synchronize()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            w1 = warm + timed
            cnn.gem_cnn_run(net, order[warm:w1], batches[warm:w1], drop[warm:w1], losses[warm:w1])
            e1.record(stream)
            stream.synchronize()
            ms = e0.elapsed_time(e1)
            lh = losses[:w1].cpu().numpy()
            pi_lo = torch.empty((pi_commits, 10), device="cuda")
            pi_hi = torch.empty((pi_commits, 10), device="cuda")
            cnn.gem_cnn_run_pi(net, order[w1:w1 + 1], batches[w1:w1 + 1], drop[w1:w1 + 1], pi_lo[:1], pi_hi[:1])
            e0.record(stream)   # the first call allocated the factor rows and select scratch
            cnn.gem_cnn_run_pi(net, order[w1 + 1:], batches[w1 + 1:], drop[w1 + 1:], pi_lo[1:], pi_hi[1:])
            e1.record(stream)
            stream.synchronize()
            ms_pi = e0.elapsed_time(e1)
            med = pi_lo.cpu().numpy()[-100:].mean(axis=0)
            cnn.gem_cnn_destroy(net)
            G.close()
        out[name] = {"commits_per_s": round(timed / (ms * 1e-3), 1), "ms": round(ms, 3),
                     "commits": timed, "workers": n, "batch": b, "params": P,
                     "loss_first_100": round(float(lh[:100].mean()), 4),
                     "loss_last_100": round(float(lh[-100:].mean()), 4),
                     "with_pi_medians": {"commits_per_s": round((pi_commits - 1) / (ms_pi * 1e-3), 1),
                                         "commits": pi_commits - 1,
                                         "median_pi_per_tensor_last_100": [round(float(v), 5) for v in med]}}
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["gem", "reference"], default="gem")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-mlp", action="store_true")
    ap.add_argument("--no-rules", action="store_true", help="skip timing the other commit rules")
    ap.add_argument("--no-flat", action="store_true", help="skip the flat P=1.2M single-commit run")
    ap.add_argument("--no-single", action="store_true", help="skip the single commits at the full size")
    ap.add_argument("--only", choices=["all", "commit", "mlp", "cnn"], default="all",
                    help="profiling aid: run only the commit batches, the async MLP or CNN runs")
    ap.add_argument("--mlp-workload", default="",
                    help="profiling aid: run only the MLP workload with this name")
    ap.add_argument("--mlp-commits", type=int, default=0,
                    help="profiling aid: timed commits per MLP workload (0: the defaults)")
    # smaller cases for profiling; the defaults are the benchmark workload
    ap.add_argument("--P", type=int, default=P_FULL)
    ap.add_argument("--workers", type=int, default=N_WORKERS)
    ap.add_argument("--batch", type=int, default=K_BATCH)
    ap.add_argument("--pool", type=int, default=POOL_ROWS)
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "gem":
        print("note: fewer than 3 warm-up steps", file=sys.stderr)
    world, rank, local, pg = dist_setup()
    if args.impl == "reference":
        run_reference(args, world, rank, pg)
    else:
        from paper_1805_08469_gb300._build import build_library
        build_library()
        if args.only in ("mlp", "cnn"):
            import torch
            torch.cuda.set_device(local)
            if args.only == "mlp":
                out = {"async_mlp": run_mlp_workloads(args, seed_offset=rank)}
            else:
                out = {"async_cnn": run_cnn_workloads(args, seed_offset=rank)}
            if rank == 0:
                print(json.dumps({"impl": "gem", "only": args.only, **out}), flush=True)
        else:
            if args.only == "commit":
                args.no_mlp = True
                args.no_flat = True
                args.no_rules = True
                args.no_single = True
            run_gem(args, world, rank, local, pg)
    if pg is not None:
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
