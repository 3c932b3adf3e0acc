"""Benchmark of the GreedyLore compression step on GB300.

Workload: the ResNet conv-gradient stack (8 layer matrices 64x576 ... 512x4608, fp32 gradients,
N=8 simulated nodes, r=8, refresh every 50 steps, MSGD), synthetic seeded gradients.  A step is
one GreedyLore iteration (Algorithm 3) over every layer matrix; the timed region covers K
consecutive steps of the real schedule, so refresh steps are included at their natural
frequency (one per tau steps).  Inputs (two alternating gradient sets of 200 MB each plus the
200 MB error state) are larger than the 129 MB L2.

Prints ONE JSON line.  `--impl reference` times the CPU oracle instead (on the host cores).
Multi-GPU (torchrun): every rank runs its own replica of the workload (the matrices are
independent and the node axis is simulated on the device), barrier + max over ranks.
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
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import workloads as W  # noqa: E402

METRIC = "gradient elems/s per GreedyLore step & % HBM roofline; subspace refresh ms"
UNIT = "grad-elem/s"
WORKLOAD = "cfg2_resnet"


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def tensor_peak_tflops():
    """The measured sustained dense bf16 tensor rate (the refresh runs inside a long step), else
    the fallback figure."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        if "bf16_tflops_sustained" in p:
            return float(p["bf16_tflops_sustained"]), "measured"
    return 1700.0, "fallback"


def refresh_flops(cfg, basis_rank):
    """Algorithmic flops of one truncated-basis refresh of every matrix: q block power iterations,
    each a pass of Mbar^T Q and of Mbar Z (2 m' n' k flops apiece), and the Rayleigh-Ritz pass
    (2 m' n' k); the k x k work is negligible beside them."""
    return sum((2 * cfg.power_iters + 1) * 2 * min(m, n) * max(m, n) * basis_rank for (m, n) in cfg.shapes)


def algorithmic_bytes(cfg, e_zero: bool):
    """Bytes a GreedyLore step must move: per node-element G (gsize) + E read/write (8 B; no
    read after an error reset); per matrix element the optimizer state (MSGD 16 B, Adam 24 B)."""
    g = 4 if cfg.grad_dtype == "f32" else 2
    per_node = g + (4 if e_zero else 8)
    opt = 16 if cfg.optimizer == "msgd" else 24
    elems = cfg.matrix_elems()
    return cfg.N * elems * per_node + elems * opt


class ClockSampler:
    """nvidia-smi samples (200 ms) of SM clock, power and throttle reasons during a region."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
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
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for nm, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


def make_handles(glr, cfg, basis_rank):
    hs = []
    for li, (m, n) in enumerate(cfg.shapes):
        hs.append(glr.GreedyLore(m, n, cfg.r, cfg.N, tau=cfg.tau, optimizer=cfg.optimizer, lr=cfg.lr,
                                 beta1=cfg.beta1, beta2=cfg.beta2, eps=cfg.eps, seed=9000 + li,
                                 basis_rank=basis_rank, power_iters=cfg.power_iters,
                                 grad_dtype=cfg.grad_dtype))
    return hs


def run_steps(hs, gsets, X, t0, K):
    import paper_2507_08784_gb300 as glr
    for s in range(K):
        glr.glr_step_group(hs, gsets[(t0 + s) % len(gsets)], X)


def timed(torch, fn):
    st = torch.cuda.current_stream()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record(st)
    fn()
    b.record(st)
    torch.cuda.synchronize()
    return a.elapsed_time(b)


def timed_steps(torch, hs, gsets, X, t0, K):
    """K steps with a CUDA event after each one (events on the launching stream); returns the
    total and the per-step milliseconds."""
    st = torch.cuda.current_stream()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(K + 1)]
    torch.cuda.synchronize()
    evs[0].record(st)
    for s in range(K):
        run_steps(hs, gsets, X, t0 + s, 1)
        evs[s + 1].record(st)
    torch.cuda.synchronize()
    per = [evs[s].elapsed_time(evs[s + 1]) for s in range(K)]
    return evs[0].elapsed_time(evs[K]), per


def bench_mode(torch, glr, cfg, prob, basis_rank, K, Wm, dist_ctx, gsets):
    """Time K steps (after Wm warm-up steps) for one basis mode; returns a dict."""
    hs = make_handles(glr, cfg, basis_rank)
    X = [torch.zeros(m, n, device="cuda") for (m, n) in cfg.shapes]
    run_steps(hs, gsets, X, 0, Wm)
    torch.cuda.synchronize()
    l0 = sum(h.stats()["launches"] for h in hs)
    t_first = Wm
    dist_ctx.barrier()
    ms, per = timed_steps(torch, hs, gsets, X, t_first, K)
    ms = dist_ctx.max(ms)
    is_ref = [(t_first + s) % cfg.tau == 0 for s in range(K)]
    nonref = [p for p, f in zip(per, is_ref) if not f]
    ref = [p for p, f in zip(per, is_ref) if f]
    nonref_ms = statistics.median(nonref) if nonref else None
    refresh_step_ms = statistics.mean(ref) if ref else None
    launches = sum(h.stats()["launches"] for h in hs) - l0
    refreshes = sum(1 for t in range(t_first, t_first + K) if t % cfg.tau == 0)
    # second pass with per-phase CUDA events (same schedule continued) for the kernel breakdown
    for h in hs:
        h.profile(True)
        h.profile_read(reset=True)
    t2 = t_first + K
    ms_prof = timed(torch, lambda: run_steps(hs, gsets, X, t2, K))
    phases = {}
    for h in hs:
        for name, v in h.profile_read(reset=True).items():
            agg = phases.setdefault(name, {"ms": 0.0, "launches": 0, "count": 0})
            for key in agg:
                agg[key] += v[key]
        h.profile(False)
    e_zero_steps = sum(1 for t in range(t2, t2 + K) if t % cfg.tau == 1)
    compose_bytes = (K * cfg.N * cfg.matrix_elems() * ((4 if cfg.grad_dtype == "f32" else 2) + 8)
                     - e_zero_steps * cfg.N * cfg.matrix_elems() * 4)
    refresh_in_prof = sum(1 for t in range(t2, t2 + K) if t % cfg.tau == 0)
    for h in hs:
        h.close()
    return {"ms": ms, "launches": launches, "refreshes": refreshes, "ms_prof": ms_prof,
            "phases": phases, "compose_bytes": compose_bytes, "refresh_in_prof": refresh_in_prof,
            "nonrefresh_step_ms": nonref_ms, "refresh_step_ms": refresh_step_ms}


def bench_e2e(torch, glr, cfg, K, Wm, dist_ctx):
    """Same metric through glr_step_group_host: every step copies the N pinned host gradients
    of every matrix in (on per-matrix copy streams, double-buffered so they overlap the previous
    step's compute) and the updated X of every matrix out to pinned host memory, inside the
    timed region, which ends with a device synchronise."""
    prob = W.make_problem(cfg)
    hs = make_handles(glr, cfg, cfg.basis_rank)
    host = [[g.cpu().pin_memory() for g in W.gradients_torch(prob, li, 0)] for li in range(len(cfg.shapes))]
    X = [torch.zeros(m, n, device="cuda") for (m, n) in cfg.shapes]
    Xh = [torch.zeros(m, n).pin_memory() for (m, n) in cfg.shapes]

    def go(k):
        for _ in range(k):
            glr.glr_step_group_host(hs, host, X, Xh)

    go(Wm)
    dist_ctx.barrier()
    ms = dist_ctx.max(timed(torch, lambda: go(K)))
    for h in hs:
        h.close()
    gsz = 4 if cfg.grad_dtype == "f32" else 2
    h2d = cfg.N * cfg.matrix_elems() * gsz
    return {"ms": ms, "h2d": h2d, "d2h": cfg.matrix_elems() * 4, "link_gbs": h2d_link_gbs(torch, h2d)}


def h2d_link_gbs(torch, nbytes, reps=3):
    """This machine's host-to-device copy rate for one step's worth of gradient bytes: one pinned
    buffer copied to the device in a single copy, best of `reps` (CUDA events)."""
    src = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    dst = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    best = float("inf")
    for _ in range(reps + 1):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        dst.copy_(src, non_blocking=True)
        e1.record()
        torch.cuda.synchronize()
        best = min(best, e0.elapsed_time(e1))
    return nbytes / (best / 1e3) / 1e9


def cpu_oracle_sample(cfg, budget_s=25.0, compressed_steps=20):
    """The oracle as it stands on the host cores: one refresh step and up to `compressed_steps`
    compressed steps of every layer matrix; the per-step time over a tau-step period is
    t_refresh + (tau - 1) * t_compressed."""
    from oracle import greedylore as O
    prob = W.make_problem(cfg)
    orcs = [O.GreedyLoreOracle(m, n, cfg.r, cfg.N, cfg.tau, optimizer=cfg.optimizer, lr=cfg.lr,
                               beta1=cfg.beta1, beta2=cfg.beta2, eps=cfg.eps, seed=9000 + li,
                               basis_rank=cfg.basis_rank)
            for li, (m, n) in enumerate(cfg.shapes)]
    Xs = [np.zeros(s) for s in cfg.shapes]
    grads = [W.gradients_numpy(prob, li, 0) for li in range(len(cfg.shapes))]
    t0 = time.perf_counter()
    for li, o in enumerate(orcs):
        Xs[li], _ = o.step(grads[li], Xs[li])
    t_refresh = time.perf_counter() - t0
    done, t_comp = 0, 0.0
    while done < compressed_steps and t_refresh + t_comp < budget_s:
        t0 = time.perf_counter()
        for li, o in enumerate(orcs):
            Xs[li], _ = o.step(grads[li], Xs[li])
        t_comp += time.perf_counter() - t0
        done += 1
    per_comp = t_comp / max(done, 1)
    per_step = (t_refresh + (cfg.tau - 1) * per_comp) / cfg.tau
    elems = cfg.N * cfg.matrix_elems()
    return {"value": elems / per_step, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"fp64 numpy oracle, all {len(cfg.shapes)} matrices: 1 refresh step "
                      f"({t_refresh:.2f} s) + {done} compressed steps ({per_comp:.2f} s each), per-step time "
                      f"over one tau={cfg.tau} period; numpy BLAS on all host cores",
            "seconds": t_refresh + t_comp}


class DistCtx:
    """One rank per GPU (torchrun's RANK / WORLD_SIZE / LOCAL_RANK / MASTER_*): NCCL on GPUs, gloo
    when the process has no GPU (the host-side tests of the multi-rank path).  Only the barrier
    and the max of the ranks' timings cross ranks; the data path has no collective."""

    def __init__(self, backend=None):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.backend = backend
        self.pg = None

    def init(self, torch):
        if self.world > 1:
            import torch.distributed as dist
            if self.backend is None:
                self.backend = "nccl" if torch.cuda.is_available() else "gloo"
            if self.backend == "nccl":
                dist.init_process_group("nccl", device_id=torch.device("cuda", self.local))
            else:
                dist.init_process_group(self.backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, v):
        if not self.pg:
            return v
        import torch
        t = torch.tensor([v], device="cuda" if self.backend == "nccl" else "cpu", dtype=torch.float64)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())


def job_rate(world, units_per_rank, ms_max):
    """Whole-job throughput of `world` replicas (weak scaling): every rank processed
    units_per_rank inside its timed region, and the job took as long as its slowest rank."""
    return world * units_per_rank / (ms_max / 1e3)


def run_reference(args):
    ctx = DistCtx()
    if ctx.world > 1 and ctx.rank != 0:
        return 0
    cfg = W.config(WORKLOAD)
    from oracle import greedylore as O
    prob = W.make_problem(cfg)
    li_order = list(range(len(cfg.shapes)))
    orcs = [O.GreedyLoreOracle(m, n, cfg.r, cfg.N, cfg.tau, optimizer=cfg.optimizer, lr=cfg.lr, beta1=cfg.beta1,
                               seed=9000 + li, basis_rank=cfg.basis_rank) for li, (m, n) in enumerate(cfg.shapes)]
    Xs = [np.zeros(s) for s in cfg.shapes]
    grads = [W.gradients_numpy(prob, li, 0) for li in li_order]

    def one_step():
        for li in li_order:
            Xs[li], _ = orcs[li].step(grads[li], Xs[li])

    for _ in range(args.warmup):
        one_step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        one_step()
    el = time.perf_counter() - t0
    elems = cfg.N * cfg.matrix_elems()
    value = elems * args.steps / el
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * el / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": WORKLOAD, "basis_rank": cfg.basis_rank,
                                            "matrices": len(cfg.shapes), "N": cfg.N, "r": cfg.r, "tau": cfg.tau},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                             "sample": f"{args.steps} consecutive oracle steps over all matrices (schedule "
                                       f"from t={args.warmup}), numpy BLAS on the host cores"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--only-headline", action="store_true",
                    help="time the truncated-basis steps only (no paper-exact pass, no e2e, no CPU baseline)")
    ap.add_argument("--e2e-steps", type=int, default=10)
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        return run_reference(args)

    import torch
    import paper_2507_08784_gb300 as glr

    ctx = DistCtx()
    torch.cuda.set_device(ctx.local)
    ctx.init(torch)
    glr.load()
    cfg = W.config(WORKLOAD)
    prob = W.make_problem(cfg)
    gsets = [[W.gradients_torch(prob, li, t) for li in range(len(cfg.shapes))] for t in range(2)]
    torch.cuda.synchronize()
    hbm_peak, peak_kind = _peaks()

    with ClockSampler(ctx.local) as clk:
        main_run = bench_mode(torch, glr, cfg, prob, cfg.basis_rank, args.steps, args.warmup, ctx, gsets)
    exact_run = None if args.only_headline else bench_mode(torch, glr, cfg, prob, 0, args.steps, args.warmup, ctx, gsets)
    e2e = None if args.only_headline else bench_e2e(torch, glr, cfg, args.e2e_steps, args.warmup, ctx)

    K = args.steps
    elems = cfg.N * cfg.matrix_elems()
    value = job_rate(ctx.world, elems * K, main_run["ms"])
    ph = main_run["phases"]
    # the refresh phase runs on one side stream per matrix, concurrently: its summed event time
    # is not wall time, so the dominant phase is taken among the phases on the step's stream and
    # the refresh's wall cost per step is added from the per-step timings
    dominant = max((k for k in ph if k != "refresh"), key=lambda k: ph[k]["ms"])
    compose = ph["compose"]
    compose_gbs = main_run["compose_bytes"] / (compose["ms"] / 1e3) / 1e9 if compose["ms"] else None
    nonrefresh_ms = main_run["nonrefresh_step_ms"]
    refresh_extra_ms = (main_run["refresh_step_ms"] - nonrefresh_ms) if main_run["refresh_step_ms"] else None
    step_bytes = algorithmic_bytes(cfg, False)
    traffic = None
    tr_path = os.path.join(ROOT, "profiles", "compose_cfg2_traffic.json")
    if os.path.exists(tr_path):
        # the DRAM bytes of one captured compose launch, valid while the kernel source is unchanged
        with open(tr_path) as f:
            rec = json.load(f)
        src = os.path.join(ROOT, "paper_2507_08784_gb300", "csrc", "k_mma.cu")
        with open(src, "rb") as f:
            if hashlib.sha256(f.read()).hexdigest() == rec.get("k_mma_cu_sha256"):
                traffic = rec.get("bytes_per_launch")
    compose_launch_bytes = main_run["compose_bytes"] / compose["launches"] if compose["launches"] else None
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ctx.world, "steps": K, "warmup": args.warmup,
        "ms_per_step": main_run["ms"] / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32", "data": "synthetic",
        "config": {"workload": WORKLOAD, "matrices": len(cfg.shapes), "shapes": "64x576..512x4608 (x2 each)",
                   "N": cfg.N, "r": cfg.r, "basis_rank": cfg.basis_rank, "tau": cfg.tau, "optimizer": cfg.optimizer,
                   "grad_dtype": cfg.grad_dtype, "refreshes_in_timed_steps": main_run["refreshes"],
                   "l2": "inputs larger than L2 (two alternating 200 MB gradient sets + 200 MB error state)",
                   "parallelism": f"replicas x{ctx.world} (node axis simulated on each GPU)"},
        "roofline": {"kernel": "compose (K1)", "bound": "hbm", "achieved": compose_gbs, "peak": hbm_peak,
                     "unit": "GB/s", "frac": (compose_gbs / hbm_peak) if compose_gbs else None,
                     "traffic": traffic, "peak_kind": peak_kind,
                     "algorithmic_bytes_per_launch_avg": compose_launch_bytes,
                     "launches_per_step": compose["launches"] / K,
                     "timing": "CUDA events around each compose launch on its stream, second timed pass of K steps",
                     "dominant_phase": dominant},
        "step_roofline": {"algorithmic_bytes_per_step": step_bytes,
                          "nonrefresh_step_ms_median": nonrefresh_ms,
                          "achieved_gbs_nonrefresh": step_bytes / (nonrefresh_ms / 1e3) / 1e9,
                          "frac_nonrefresh": step_bytes / (nonrefresh_ms / 1e3) / 1e9 / hbm_peak,
                          "grad_elems_per_s_nonrefresh": elems / (nonrefresh_ms / 1e3)},
        "refresh_ms_all_matrices": refresh_extra_ms,
        "refresh_wall_ms_per_step": (refresh_extra_ms * main_run["refreshes"] / K) if refresh_extra_ms else None,
        "refresh_ms_per_layer": refresh_extra_ms / len(cfg.shapes) if refresh_extra_ms else None,
        "refresh_tensor": None if not refresh_extra_ms else {
            "flops": refresh_flops(cfg, cfg.basis_rank),
            "tflops": refresh_flops(cfg, cfg.basis_rank) / (refresh_extra_ms / 1e3) / 1e12,
            "frac_of_tensor_peak": refresh_flops(cfg, cfg.basis_rank) / (refresh_extra_ms / 1e3) / 1e12
                                   / tensor_peak_tflops()[0],
            "peak": tensor_peak_tflops()[0], "peak_kind": tensor_peak_tflops()[1] + " bf16 sustained",
            "note": "the truncated refresh runs on the FP32 pipes; bound by HBM and latency, not the tensor cores"},
        "phases_ms_per_step": {k: v["ms"] / K for k, v in ph.items()},
        "phases_note": "refresh = summed event time of the concurrent per-matrix refresh streams",
        "phase_launches": {k: v["launches"] for k, v in ph.items()},
        "paper_exact_basis": None if exact_run is None else {
            "value": job_rate(ctx.world, elems * K, exact_run["ms"]),
            "ms_per_step": exact_run["ms"] / K,
            "nonrefresh_step_ms_median": exact_run["nonrefresh_step_ms"],
            "refresh_ms_all_matrices": (exact_run["refresh_step_ms"] - exact_run["nonrefresh_step_ms"])
            if exact_run["refresh_step_ms"] else None,
            "phases_ms_per_step": {k: v["ms"] / K for k, v in exact_run["phases"].items()}},
        "e2e": None if e2e is None else {"value": job_rate(ctx.world, elems * args.e2e_steps, e2e["ms"]), "unit": UNIT,
                                         "h2d_bytes_per_step": e2e["h2d"], "d2h_bytes_per_step": e2e["d2h"],
                                         "h2d_link_gbs": e2e["link_gbs"],
                                         "frac_of_link": (e2e["h2d"] / (e2e["ms"] / args.e2e_steps / 1e3) / 1e9)
                                                         / e2e["link_gbs"]},
        "gpu_launches": main_run["launches"],
        "clocks": clk.summary(),
    }
    if ctx.rank == 0 and ctx.world == 1 and not args.no_cpu_baseline and not args.only_headline:
        line["cpu_baseline"] = cpu_oracle_sample(cfg)
    if ctx.rank == 0:
        print(json.dumps(line))
    if ctx.pg:
        ctx.pg.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
