"""Benchmark of the GreedyLore compression step on GB300.

Headline workload: the 8-layer d = 4096 / ffn = 11008 decoder stack (56 layer matrices: Wq, Wk,
Wv, Wo 4096 x 4096, Wgate, Wup 11008 x 4096, Wdown 4096 x 11008), N = 4 simulated nodes, bf16
gradients, fp32 error state, r = 128 with a truncated basis of k = 256, Adam, refresh every 200
steps; seeded synthetic low-rank-plus-noise gradients of those shapes.  A step is one GreedyLore
iteration (Algorithm 3) over every matrix of the stack through glr_step_group; the timed region
covers K consecutive steps of the real schedule.  The refresh (Semi-Lazy SVD) is also timed on its
own: every handle is forced to refresh (glr_refresh) and that step is timed, three times.  Inputs
(two alternating 13 GB gradient sets and the 26 GB error state) are far larger than the 129 MB L2.
The ResNet conv stack (fp32, r = 8) and the d = 2048 decoder stack (bf16, r = 32) are timed as
extra keys.

Prints ONE JSON line.  `--impl reference` times the CPU oracle instead (on the host cores).
Multi-GPU (torchrun): every rank runs its own replica of the workload (the matrices are
independent and the node axis is simulated on the device), barrier + max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import dataclasses
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
WORKLOAD = "cfg5_llama_d4096"
EXTRA_WORKLOADS = ("cfg2_resnet", "cfg3_llama_d2048", "cfg4_refresh")
PAPER_EXACT = "cfg5_layer_paper_exact"     # one d = 4096 decoder layer with the full m' x m' basis


def paper_exact_config():
    """One layer of the d = 4096 decoder stack (Wq, Wk, Wv, Wo, Wgate, Wup, Wdown; N = 4, bf16,
    Adam, r = 128) with basis_rank = 0: the paper-exact basis of Eq. SVD-P1, refreshed by the
    blocked Jacobi eigen-solve, its scores the dense U^T Mbar."""
    base = W.config("cfg5_llama_d4096")
    return dataclasses.replace(base, name=PAPER_EXACT, shapes=base.shapes[:7], basis_rank=0)


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


TF32_OVER_BF16 = 1.1 / 2.25     # nominal dense TF32 / BF16 tensor rates (the refresh products are TF32)


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


def refresh_mode_of(cfg):
    """The refresh-stress workload (tau = 1) runs Algorithm 4: a refresh every step that still
    compresses with the new basis (under Algorithm 3 every step would go uncompressed)."""
    return "alg4" if cfg.tau == 1 else "alg3"


def make_handles(glr, cfg, basis_rank):
    hs = []
    for li, (m, n) in enumerate(cfg.shapes):
        hs.append(glr.GreedyLore(m, n, cfg.r, cfg.N, tau=cfg.tau, refresh_mode=refresh_mode_of(cfg),
                                 optimizer=cfg.optimizer, lr=cfg.lr,
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


def compose_bytes(cfg, compressed_steps, reset_steps):
    """Algorithmic bytes of the compose launches (K1): per node-element the gradient and the error
    state read + write (no read right after an error reset), per matrix element the Mbar write."""
    g = 4 if cfg.grad_dtype == "f32" else 2
    per = cfg.N * cfg.matrix_elems() * (g + 8) + cfg.matrix_elems() * 4
    return compressed_steps * per + reset_steps * (per - cfg.N * cfg.matrix_elems() * 4)


def bench_mode(torch, glr, cfg, basis_rank, K, Wm, dist_ctx, gsets, refresh_reps=0):
    """Time K steps (after Wm warm-up steps) of the real schedule; then the same K steps again with
    per-phase CUDA events; then `refresh_reps` forced refresh steps.  Returns a dict."""
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
    resets = sum(1 for t in range(t2, t2 + K) if t % cfg.tau == 1)
    comp_bytes = compose_bytes(cfg, K - resets, resets)
    # the refresh on its own: every handle forced to refresh at the next step, that step timed
    forced = []
    t3 = t2 + K
    for rep in range(refresh_reps):
        for h in hs:
            h.refresh()
        forced.append(timed(torch, lambda: run_steps(hs, gsets, X, t3, 1)))
        t3 += 1
        run_steps(hs, gsets, X, t3, 1)             # the step after (error reset), untimed
        t3 += 1
    path = hs[0].stats()["path"]
    sweeps = [h.stats()["last_refresh_sweeps"] for h in hs]
    for h in hs:
        h.close()
    return {"ms": ms, "launches": launches, "refreshes": refreshes, "ms_prof": ms_prof, "phases": phases,
            "compose_bytes": comp_bytes, "nonrefresh_step_ms": statistics.median(nonref) if nonref else None,
            "refresh_step_ms_in_window": statistics.mean(ref) if ref else None,
            "forced_refresh_step_ms": forced, "path": path, "sweeps": sweeps}


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
    del host, Xh, X
    return {"ms": ms, "h2d": h2d, "d2h": cfg.matrix_elems() * 4, "link_gbs": h2d_link_gbs(torch, min(h2d, 1 << 30))}


def h2d_link_gbs(torch, nbytes, reps=3):
    """This machine's host-to-device copy rate: one pinned buffer copied to the device in a single
    copy, best of `reps` (CUDA events)."""
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


def oracle_sample_step(cfg, li, nodes, t=1):
    """One compressed step of the CPU oracle on layer matrix li with `nodes` nodes, timed: the
    oracle as it stands, started from Algorithm 3's input basis U = I with the refresh step
    behind it (t = 1), so it runs the compressed path (Approx-Top-r, projection, error feedback,
    optimizer).  Returns (seconds, node-elements processed)."""
    from oracle import greedylore as O
    one = W.config(cfg.name, shapes=cfg.shapes[: li + 1])      # layer li's factors only
    prob = W.make_problem(one)
    m, n = cfg.shapes[li]
    o = O.GreedyLoreOracle(m, n, cfg.r, nodes, cfg.tau, optimizer=cfg.optimizer, lr=cfg.lr, beta1=cfg.beta1,
                           beta2=cfg.beta2, eps=cfg.eps, seed=9000 + li, basis_rank=cfg.basis_rank)
    o.t = t
    G = W.gradients_numpy(prob, li, t, workers=list(range(nodes)))
    t0 = time.perf_counter()
    o.step(G, np.zeros((m, n)))
    return time.perf_counter() - t0, nodes * m * n


def cpu_oracle_sample(cfg):
    """The oracle as it stands on the host cores, on a bounded sample of the workload: one
    compressed step of the stack's square matrix (the shape of 32 of its 56 matrices) with all N
    nodes, numpy BLAS on every core; and the same step with one node in a single-threaded process."""
    li = 0
    secs, units = oracle_sample_step(cfg, li, cfg.N)
    m, n = cfg.shapes[li]
    out = {"value": units / secs, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
           "sample": f"one compressed step of one {m}x{n} matrix of the stack with all {cfg.N} nodes "
                     f"({secs:.2f} s; fp64 numpy oracle from U = I, BLAS on every host core); the rate is "
                     f"node-elements per second on that shape", "seconds": secs}
    code = ("import sys; sys.path.insert(0, %r); import bench, workloads as W; "
            "s, u = bench.oracle_sample_step(W.config(%r), 0, 1); print(u / s, s)") % (ROOT, cfg.name)
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    try:
        res = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=120)
        v, secs1 = (float(x) for x in res.stdout.split()[-2:])
        out["single_thread"] = {"value": v, "cores": 1, "seconds": secs1,
                                "sample": f"the same step with 1 node in one thread ({secs1:.2f} s)"}
    except Exception as e:                      # report, do not fail the benchmark
        out["single_thread"] = {"value": None, "error": str(e)[:200]}
    return out


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
    """The reference arm: the CPU oracle (fp64 numpy, the host cores), each step a bounded sample
    of the workload (one compressed step of one of the stack's square matrices, one node), the
    rate in the benchmark's unit.  Ranks other than 0 exit without work."""
    ctx = DistCtx()
    if ctx.world > 1 and ctx.rank != 0:
        return 0
    cfg = W.config(WORKLOAD)
    for _ in range(args.warmup):
        oracle_sample_step(cfg, 0, 1)
    secs, units = 0.0, 0
    for _ in range(args.steps):
        s_, u_ = oracle_sample_step(cfg, 0, 1)
        secs += s_
        units += u_
    value = units / secs
    m, n = cfg.shapes[0]
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": WORKLOAD, "basis_rank": cfg.basis_rank,
                                            "matrices": len(cfg.shapes), "N": cfg.N, "r": cfg.r, "tau": cfg.tau},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                             "sample": f"each step: one compressed oracle step of one {m}x{n} matrix of the "
                                       f"stack with one node (fp64 numpy from U = I, BLAS on the host cores)"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def traffic_record(kernel_file, record):
    """DRAM bytes per unit of one captured launch (profiles/), valid while the kernel source is
    the one that was captured."""
    path = os.path.join(ROOT, "profiles", record)
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rec = json.load(f)
    with open(os.path.join(ROOT, "paper_2507_08784_gb300", "csrc", kernel_file), "rb") as f:
        if hashlib.sha256(f.read()).hexdigest() != rec.get("source_sha256"):
            return None
    return rec


def summarize(cfg, run, K, world, hbm_peak):
    """Rate, step roofline and phase breakdown of one bench_mode run."""
    elems = cfg.N * cfg.matrix_elems()
    step_bytes = algorithmic_bytes(cfg, False)
    nonref = run["nonrefresh_step_ms"]
    ph = run["phases"]
    comp = ph.get("compose", {"ms": 0.0, "launches": 0})
    return {
        "value": job_rate(world, elems * K, run["ms"]), "ms_per_step": run["ms"] / K,
        "path": ["strip", "mma", "tcgen05", "library", "plain"][run["path"]],
        "nonrefresh_step_ms_median": nonref,
        "grad_elems_per_s_nonrefresh": elems / (nonref / 1e3) if nonref else None,
        "step_roofline": {"algorithmic_bytes_per_step": step_bytes,
                          "achieved_gbs": step_bytes / (nonref / 1e3) / 1e9 if nonref else None,
                          "frac": step_bytes / (nonref / 1e3) / 1e9 / hbm_peak if nonref else None},
        "compose_gbs": run["compose_bytes"] / (comp["ms"] / 1e3) / 1e9 if comp["ms"] else None,
        "phases_ms_per_step": {k: round(v["ms"] / K, 4) for k, v in ph.items()},
        "phase_launches_per_step": {k: v["launches"] / K for k, v in ph.items()},
    }


def bench_paper_exact(torch, glr, K, Wm, ctx, hbm_peak):
    """The paper-exact basis on one d = 4096 decoder layer: compressed steps with the dense scores
    U^T Mbar (TF32 tcgen05, 2 m'^2 n' flops per matrix) and one forced refresh step (the blocked
    Jacobi eigen-solve of Mbar Mbar^T for all 7 matrices)."""
    xc = paper_exact_config()
    xp = W.make_problem(xc)
    xs = [[W.gradients_torch(xp, li, t) for li in range(len(xc.shapes))] for t in range(2)]
    xr = bench_mode(torch, glr, xc, 0, K, Wm, ctx, xs, refresh_reps=1)
    out = summarize(xc, xr, K, ctx.world, hbm_peak)
    out["config"] = {"matrices": len(xc.shapes), "shapes": "4 x 4096x4096, 2 x 11008x4096, 4096x11008",
                     "N": xc.N, "r": xc.r, "basis_rank": 0, "tau": xc.tau, "grad_dtype": xc.grad_dtype,
                     "optimizer": xc.optimizer, "refresh_mode": refresh_mode_of(xc)}
    flops = sum(2.0 * min(m, n) ** 2 * max(m, n) for (m, n) in xc.shapes)
    lam_ms = xr["phases"]["lambda"]["ms"] / K
    tpeak, tkind = tensor_peak_tflops()
    out["scores_tensor"] = {
        "kernel": "tc_kernel<LambdaU> (U^T Mbar, v_j in the epilogue)", "flops_per_step": flops, "ms": lam_ms,
        "tflops": flops / (lam_ms / 1e3) / 1e12, "tf32_peak": tpeak * TF32_OVER_BF16,
        "frac_of_tf32_peak": flops / (lam_ms / 1e3) / 1e12 / (tpeak * TF32_OVER_BF16),
        "peak_kind": tkind + " bf16 sustained x nominal TF32/BF16 ratio (1.1 / 2.25)"}
    forced, nonref = xr["forced_refresh_step_ms"], xr["nonrefresh_step_ms"]
    ref = statistics.median(forced) - nonref if forced and nonref else None
    out["refresh"] = {"forced_refresh_step_ms": forced, "refresh_ms_per_layer": ref,
                      "refresh_ms_per_matrix": ref / len(xc.shapes) if ref else None,
                      "jacobi_sweeps": xr["sweeps"],
                      "method": "H = Mbar Mbar^T (FFMA), blocked two-sided Jacobi: 128-index pair blocks "
                                "solved by one scalar-Jacobi sweep each, block rotations as FFMA products"}
    del xs
    torch.cuda.empty_cache()
    return out


def ncu_case_exact():
    """One 4096 x 4096 matrix of the headline stack with the full basis (basis_rank = 0) for 4
    steps: step 0 is the blocked Jacobi refresh (about 15 sweeps of 63 rounds, each round one pair
    sweep launch and two block-product launches), steps 1-3 run the dense scores (LambdaU)."""
    import torch
    import paper_2507_08784_gb300 as glr
    base = W.config(WORKLOAD)
    cfg = dataclasses.replace(base, shapes=base.shapes[:1], basis_rank=0)
    prob = W.make_problem(cfg)
    gs = [W.gradients_torch(prob, 0, t) for t in range(2)]
    hs = make_handles(glr, cfg, 0)
    X = [torch.zeros(*cfg.shapes[0], device="cuda")]
    for t in range(4):
        glr.glr_step_group(hs, [gs[t % 2]], X)
    torch.cuda.synchronize()
    print(json.dumps({"ncu_case": "paper_exact", "shape": cfg.shapes[0], "N": cfg.N, "r": cfg.r,
                      "sweeps": hs[0].stats()["last_refresh_sweeps"], "path": hs[0].stats()["path"]}))
    hs[0].close()
    return 0


def ncu_case(refresh=False, stress=False):
    """One 4096 x 4096 matrix of the headline stack for 4 steps (about 1.1 GB of state): the
    compose launch of step 2 (index 2 among compose launches) is a full one; with refresh, a
    fifth step forced to refresh.  With stress: the refresh-stress matrix (4096 x 11008, N = 8,
    k = 128, Algorithm 4) for 3 steps, each a refresh (about 4 GB of state)."""
    import torch
    import paper_2507_08784_gb300 as glr
    if stress:
        cfg = W.config("cfg4_refresh")
        prob = W.make_problem(cfg)
        gs = [W.gradients_torch(prob, 0, t) for t in range(2)]
        hs = make_handles(glr, cfg, cfg.basis_rank)
        X = [torch.zeros(*cfg.shapes[0], device="cuda")]
        for t in range(3):
            glr.glr_step_group(hs, [gs[t % 2]], X)
        torch.cuda.synchronize()
        print(json.dumps({"ncu_case": "cfg4_refresh", "shape": cfg.shapes[0], "N": cfg.N, "k": cfg.basis_rank,
                          "path": hs[0].stats()["path"]}))
        hs[0].close()
        return 0
    cfg = W.config(WORKLOAD, shapes=W.config(WORKLOAD).shapes[:1])
    prob = W.make_problem(cfg)
    gs = [W.gradients_torch(prob, 0, t) for t in range(2)]
    hs = make_handles(glr, cfg, cfg.basis_rank)
    X = [torch.zeros(*cfg.shapes[0], device="cuda")]
    for t in range(4):
        glr.glr_step_group(hs, [gs[t % 2]], X)
    if refresh:                                    # then one forced refresh step
        hs[0].refresh()
        glr.glr_step_group(hs, [gs[0]], X)
    torch.cuda.synchronize()
    print(json.dumps({"ncu_case": WORKLOAD, "shape": cfg.shapes[0], "N": cfg.N,
                      "node_elems_per_compose": cfg.N * cfg.matrix_elems(), "path": hs[0].stats()["path"]}))
    hs[0].close()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--only-headline", action="store_true",
                    help="time the headline workload only (no extra workloads, no e2e, no CPU baseline)")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--refresh-reps", type=int, default=3)
    ap.add_argument("--ncu-case", nargs="?", const="steps", choices=["steps", "refresh", "stress", "exact"],
                    help="a small case for kernel captures: one 4096 x 4096 matrix of the headline stack "
                         "(N = 4, r = 128, k = 256, bf16, Adam), 4 steps: refresh, reset, then two full "
                         "steps; 'refresh' adds a fifth step forced to refresh; 'stress' runs the refresh-stress "
                         "matrix (4096 x 11008, N = 8, k = 128) for 3 refresh steps")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        return run_reference(args)
    if args.ncu_case == "exact":
        return ncu_case_exact()
    if args.ncu_case:
        return ncu_case(args.ncu_case == "refresh", args.ncu_case == "stress")

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
    K = args.steps

    with ClockSampler(ctx.local) as clk:
        main_run = bench_mode(torch, glr, cfg, cfg.basis_rank, K, args.warmup, ctx, gsets,
                              refresh_reps=args.refresh_reps)
    del gsets
    torch.cuda.empty_cache()
    e2e = None if args.only_headline else bench_e2e(torch, glr, cfg, args.e2e_steps, 3, ctx)
    extras = {}
    if not args.only_headline:
        for name in EXTRA_WORKLOADS:
            xc = W.config(name)
            xp = W.make_problem(xc)
            xs = [[W.gradients_torch(xp, li, t) for li in range(len(xc.shapes))] for t in range(2)]
            xr = bench_mode(torch, glr, xc, xc.basis_rank, K, args.warmup, ctx, xs)
            extras[name] = summarize(xc, xr, K, ctx.world, hbm_peak)
            extras[name]["config"] = {"matrices": len(xc.shapes), "N": xc.N, "r": xc.r, "basis_rank": xc.basis_rank,
                                      "tau": xc.tau, "grad_dtype": xc.grad_dtype, "optimizer": xc.optimizer,
                                      "refresh_mode": refresh_mode_of(xc)}
            if xc.tau == 1:     # every step refreshes: the step is the refresh-stress number
                rflops = refresh_flops(xc, xc.basis_rank)
                tpeak, tkind = tensor_peak_tflops()
                ms = extras[name]["ms_per_step"]
                extras[name]["refresh_every_step"] = {
                    "ms_per_step": ms, "ms_per_layer": ms / len(xc.shapes), "refresh_flops": rflops,
                    "tflops": rflops / (ms / 1e3) / 1e12, "tf32_peak": tpeak * TF32_OVER_BF16,
                    "frac_of_tf32_peak": rflops / (ms / 1e3) / 1e12 / (tpeak * TF32_OVER_BF16),
                    "peak_kind": tkind + " bf16 sustained x nominal TF32/BF16 ratio (1.1 / 2.25)"}
            del xs
            torch.cuda.empty_cache()
        extras[PAPER_EXACT] = bench_paper_exact(torch, glr, K, args.warmup, ctx, hbm_peak)

    elems = cfg.N * cfg.matrix_elems()
    head = summarize(cfg, main_run, K, ctx.world, hbm_peak)
    ph = main_run["phases"]
    comp = ph["compose"]
    comp_launch_bytes = main_run["compose_bytes"] / comp["launches"] if comp["launches"] else None
    comp_ms = comp["ms"] / comp["launches"] if comp["launches"] else None
    achieved = comp_launch_bytes / (comp_ms / 1e3) / 1e9 if comp_ms else None
    rec = traffic_record("k_tc.cu", "compose_tcgen05_traffic.json")
    traffic = None
    if rec:   # the captured launch's DRAM bytes scaled to one launch of this workload by its node-elements
        traffic = rec["dram_bytes"] * (cfg.N * cfg.matrix_elems()) / rec["node_elems"]
    nonref = main_run["nonrefresh_step_ms"]
    forced = main_run["forced_refresh_step_ms"]
    ref_step = statistics.median(forced) if forced else None
    refresh_ms = (ref_step - nonref) if (ref_step and nonref) else None
    layers = len(cfg.shapes) // 7
    amort = ((cfg.tau - 1) * nonref + ref_step) / cfg.tau if ref_step else None
    tpeak, tkind = tensor_peak_tflops()
    rflops = refresh_flops(cfg, cfg.basis_rank)
    line = {
        "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": ctx.world, "steps": K,
        "warmup": args.warmup, "ms_per_step": main_run["ms"] / K, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16 gradients, fp32 state, TF32 tensor-core products",
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "matrices": len(cfg.shapes),
                   "shapes": "8 layers x {4 x 4096x4096, 2 x 11008x4096, 4096x11008}", "N": cfg.N, "r": cfg.r,
                   "basis_rank": cfg.basis_rank, "tau": cfg.tau, "optimizer": cfg.optimizer,
                   "grad_dtype": cfg.grad_dtype, "refreshes_in_timed_steps": main_run["refreshes"],
                   "path": head["path"],
                   "l2": "inputs larger than L2 (two alternating 13 GB gradient sets + 26 GB error state)",
                   "parallelism": f"replicas x{ctx.world} (node axis simulated on each GPU)"},
        "roofline": {"kernel": "compose (K1, tcgen05)", "bound": "hbm", "achieved": achieved, "peak": hbm_peak,
                     "unit": "GB/s", "frac": (achieved / hbm_peak) if achieved else None, "traffic": traffic,
                     "peak_kind": peak_kind, "algorithmic_bytes_per_launch": comp_launch_bytes,
                     "launch_ms": comp_ms, "launches_per_step": comp["launches"] / K,
                     "timing": "CUDA events around each compose launch on its stream, second timed pass of K steps"},
        "step_roofline": head["step_roofline"],
        "grad_elems_per_s_nonrefresh": head["grad_elems_per_s_nonrefresh"],
        "nonrefresh_step_ms_median": nonref,
        "refresh": {"forced_refresh_step_ms": forced, "refresh_ms_all_matrices": refresh_ms,
                    "refresh_ms_per_layer": refresh_ms / layers if refresh_ms else None,
                    "refresh_ms_per_matrix": refresh_ms / len(cfg.shapes) if refresh_ms else None,
                    "tau_amortised_step_ms": amort,
                    "tau_amortised_value": elems / (amort / 1e3) if amort else None,
                    "tensor": None if not refresh_ms else {
                        "flops": rflops, "tflops": rflops / (refresh_ms / 1e3) / 1e12,
                        "frac_of_tensor_peak": rflops / (refresh_ms / 1e3) / 1e12 / (tpeak * TF32_OVER_BF16),
                        "peak": tpeak * TF32_OVER_BF16,
                        "peak_kind": tkind + " bf16 sustained x nominal TF32/BF16 ratio (1.1 / 2.25): the "
                                     "refresh products are TF32 tcgen05 MMAs"},
                    "how": "every handle forced to refresh (glr_refresh), that step timed with CUDA events, "
                           f"{len(forced)} repeats; refresh ms = that step minus the median compressed step"},
        "phases_ms_per_step": head["phases_ms_per_step"],
        "phase_launches_per_step": head["phase_launches_per_step"],
        "phases_note": "refresh = summed event time of the concurrent per-matrix refresh streams",
        "extra_workloads": extras,
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
