"""Benchmark: one GA generation of the E2LLM deployment search per step.

A step is the whole hot path over one population: DP_Pipe for every replica
and variant with the decode batch sweep, the objective, the elites and the
generation step (tournament, crossover + repair, mutation).  The default
workload is the largest single-GPU configuration: 512 devices, a 126-block
model, up to 64 replicas per genome, population 16,384.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

value: genome evaluations per second over the timed steps, device time with
CUDA events on the engine's stream, L2 flushed (256 MB write) between steps.
e2e: the same metric through the C ABI with pinned host buffers: each step is
one e2_run_generation_io call that uploads the population, evaluates, steps,
and reads fitness and the next population back, synchronising once.
roofline: the DP_Pipe kernel (both of its launches where the replica sizes
form two shared-memory classes) against the integer issue rate of its own
instruction mix, measured in the same run by e2_probe_int_rate.
configs: the other four workloads, device-timed the same way (the 256-device
one over 200 back-to-back generations: generations per second).
--impl reference times the CPU oracle on the host cores.  Under torchrun each
rank runs an independent replica search (its own seed) on its own GPU; value
is the sum over ranks divided by the slowest rank's time.
"""
from __future__ import annotations

import argparse
import dataclasses
import datetime
import json
import math
import os
import statistics
import subprocess
import tempfile
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2606_03770_gb300 import workloads as W  # noqa: E402

METRIC = "genome evaluations/sec (GA generations on device)"
UNIT = "genomes/s"
WORKLOAD = "c4"
OTHER_CONFIGS = ("c1_tiny", "c2", "c3", "c5")
L2_FLUSH_BYTES = 256 << 20
# algorithmic int32 operations per unit of DP work, the rule of about five
# integer operations per examined candidate: per crossover probe (of a
# bisection, or the one-step advance to the next cell) two key loads, a
# compare, a select or step and an index update; per DP cell a min, a max
# with the link key, two guards and a store.  Probes and cells are the
# kernel's own tallies (e2_get_stats).
OPS_PER_PROBE = 5
OPS_PER_CELL = 5
INT32_LANES_PER_SM = 128
# dram__bytes_read.sum + dram__bytes_write.sum of the two DP launches of one
# generation at the default workload (class 0: 30.21 + 9.29 MB, class 1:
# 24.55 + 5.46 MB), from the ncu capture in profiles/; cold (ncu flushes the
# caches before each launch), so it counts the L2-resident order-key rows
# again
DP_TRAFFIC_BYTES = 69_413_632
DP_TRAFFIC_SOURCE = "profiles/dp_eval_c4_gen2.md (dram read+write, both DP launches of one generation, cold)"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default=WORKLOAD)
    ap.add_argument("--seed", type=int, default=2026)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-configs", action="store_true", help="skip the other workloads' lines")
    ap.add_argument("--repeats", action="store_true",
                    help="instead of timing: how often replicas repeat over the workload's generations")
    ap.add_argument("--cpu-only", action="store_true",
                    help="instead of timing the GPU: the oracle's CPU baseline of the workload (all cores, one core)")
    ap.add_argument("--clocks-dir", default=tempfile.gettempdir(),
                    help="folder for the raw nvidia-smi samples of the timed region (clocks_rank<i>.csv)")
    ap.add_argument("--roles", default="bits", choices=["bits", "search"],
                    help="replica roles: bits of the genome, or Alg. 2's brute-force search")
    return ap.parse_args()


def problem(args):
    prob = W.make_config(args.config)
    if args.roles == "search":
        prob = dataclasses.replace(prob, role_search=1)
    return prob


def workload_label(prob):
    mdl = W.CONFIGS[prob.name]["model"]
    kv = f"GQA {mdl['kv_heads']} KV heads" if mdl.get("kv_heads") else "MHA"
    roles = "roles searched per genome (Alg. 2)" if prob.role_search else "one role bit per replica"
    return (f"{prob.name}: M={prob.M} devices, N={prob.N} blocks (d={mdl['d']}, ffn={mdl['ffn']}, {kv}, "
            f"{mdl['wbits']}-bit weights), K_max={prob.K_max} replicas, P={prob.P}, Q={prob.Q}, "
            f"b_max={prob.b_max}, {roles}, one generation per step"
            + (", congestion redrawn per generation" if prob.redraw else ""))


def dist_info():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def max_over_ranks(x, world, device="cpu"):
    """Largest value of x over the ranks (the slowest replica's time)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(units_per_rank, world, t_max):
    """Whole-job throughput of `world` independent replicas that each processed
    `units_per_rank` units, the slowest in t_max seconds (weak scaling)."""
    return units_per_rank * world / t_max


class Clocks:
    """nvidia-smi sampling around the timed region.  Samples carry the host
    wall clock at which they were read; those inside the region's window are
    kept (the one nearest to it when the region is shorter than the sampling
    interval, marked "nearest")."""
    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, index, folder):
        self.index = index
        self.proc = None
        self.path = os.path.join(folder, f"clocks_rank{index}.csv")
        self.t0 = self.t1 = None

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "20"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
            return
        deadline = time.time() + 10.0            # wait for the sampler's first line
        while time.time() < deadline and self.proc.poll() is None:
            if os.path.getsize(self.path) > 0:
                break
            time.sleep(0.01)

    def begin(self):
        self.t0 = time.time()

    def end(self):
        self.t1 = time.time()

    def _rows(self):
        for line in open(self.path):
            p = [x.strip() for x in line.split(",")]
            if len(p) < 10:
                continue
            try:
                ts = datetime.datetime.strptime(p[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                yield ts, float(p[2]), float(p[3]), [n for n, v in zip(self.NAMES, p[6:10]) if v.lower() == "active"]
            except ValueError:
                continue

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        rows = list(self._rows())
        if not rows or self.t0 is None:
            return None
        inside = [r for r in rows if self.t0 <= r[0] <= self.t1]
        kept, how = inside, "inside the timed region"
        if not inside:
            mid = 0.5 * (self.t0 + self.t1)
            kept, how = [min(rows, key=lambda r: abs(r[0] - mid))], "nearest to the timed region"
        reasons = sorted({n for r in kept for n in r[3]})
        return {"sm_mhz": statistics.median(r[1] for r in kept), "sm_max_mhz": max(r[2] for r in kept),
                "reasons": reasons, "samples": len(kept), "window": how,
                "timed_region_s": self.t1 - self.t0}


def _oracle_eval_rate(prob, pop, sample, nthreads):
    """Seconds the oracle takes to evaluate `sample` genomes on `nthreads` threads."""
    from oracle import oracle as O
    sub = {k: np.ascontiguousarray(v[:sample]) for k, v in pop.items()}
    op = O.OracleProblem(prob)
    t0 = time.perf_counter()
    op.eval_population(sub, prob.K_max, nthreads=nthreads)
    return time.perf_counter() - t0


def cpu_baseline(prob, seed, budget_s=30.0):
    """The oracle, as it is, on this host's cores: a bounded sample of one
    generation's genomes evaluated on every core and on one core, each scaled
    to the population, plus the elites and generation step of the full
    population.  The sample grows from a few genomes per thread until it takes
    about a third of the budget."""
    from oracle import oracle as O
    ga = O.ga_of(prob)
    pop = O.init_population(ga, seed)
    nt = O.num_threads()
    sample, t_eval = nt, _oracle_eval_rate(prob, pop, min(prob.P, nt), nt)
    while sample < prob.P and t_eval < budget_s / 6:
        grow = min(prob.P, sample * 4)
        sample, t_eval = grow, _oracle_eval_rate(prob, pop, grow, nt)
    one = 1
    t_one = _oracle_eval_rate(prob, pop, 1, 1)
    while one < prob.P and t_one < budget_s / 6:
        grow = min(prob.P, one * 4)
        one, t_one = grow, _oracle_eval_rate(prob, pop, grow, 1)
    full_fit = np.zeros((prob.P, 4))
    full_fit[:, 0] = np.arange(prob.P, dtype=np.float64)      # any order; only timing matters here
    t0 = time.perf_counter()
    e = O.elites(ga, pop, full_fit)
    O.ga_step(ga, seed, 1, pop, full_fit, e)
    t_ga = time.perf_counter() - t0
    t_gen = t_eval * prob.P / sample + t_ga
    t_gen1 = t_one * prob.P / one + t_ga
    return {"value": prob.P / t_gen, "unit": UNIT, "cores": nt, "kind": "oracle",
            "sample": f"{sample} of {prob.P} genomes of one generation evaluated on {nt} threads "
                      f"({t_eval:.2f} s), scaled to the population, plus the elites and generation "
                      f"step of the full population ({t_ga:.3f} s)",
            "single_core": {"value": prob.P / t_gen1, "unit": UNIT, "cores": 1,
                            "sample": f"{one} genomes on one thread ({t_one:.2f} s), scaled to the "
                                      f"population, plus the same elites and generation step"}}


def run_reference(args):
    rank, world, _ = dist_info()
    if rank != 0:
        return
    prob = problem(args)
    from oracle import oracle as O
    nt = O.num_threads()
    ga = O.ga_of(prob)
    pop = O.init_population(ga, args.seed)
    op = O.OracleProblem(prob)
    # per step, a bounded sample: a few genomes per thread, sized so that one
    # step's evaluation takes about 5 s of host time
    t_probe = _oracle_eval_rate(prob, pop, min(prob.P, nt), nt)
    sample = max(1, min(prob.P, int(min(prob.P, nt) * 5.0 / max(t_probe, 1e-3))))
    times, walls = [], []
    fit = np.zeros((prob.P, 4))
    for step in range(args.warmup + args.steps):
        w0 = time.perf_counter()
        sub = {k: np.ascontiguousarray(v[(step * sample) % prob.P:][:sample]) for k, v in pop.items()}
        n = len(sub["nclus"])
        t0 = time.perf_counter()
        out = op.eval_population(sub, prob.K_max, nthreads=nt)
        t_eval = time.perf_counter() - t0
        fit[:] = 0.0
        fit[:n] = out["fitness"]
        t0 = time.perf_counter()
        e = O.elites(ga, pop, fit)
        nxt = O.ga_step(ga, args.seed, step + 1, pop, fit, e)
        t_ga = time.perf_counter() - t0
        pop = nxt
        if step >= args.warmup:
            times.append(t_eval * prob.P / n + t_ga)      # one generation of P genomes, scaled
            walls.append(time.perf_counter() - w0)
    t = sum(times)
    value = prob.P * len(times) / t
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t / len(times),
            "ms_per_step_is": "a full generation of P genomes, scaled from the sample evaluated per step",
            "wall_ms_per_step_measured": 1e3 * sum(walls) / len(walls),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded fleet, links and dense-decoder profile)",
            "config": {"workload": workload_label(prob), "sample_genomes_per_step": sample},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": nt, "kind": "oracle",
                             "sample": f"per step, {sample} of {prob.P} genomes evaluated by the oracle on "
                                       f"{nt} threads and scaled to the population, plus the elites and "
                                       f"generation step of the full population"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def int_peak(torch, stream, clocks_dir, index):
    """The DP's instruction mix (min, max, compare, select, add) at full
    occupancy, through e2_probe_int_rate: operations per second, and per SM
    per clock at the SM clock sampled during the probe launches."""
    from paper_2606_03770_gb300 import e2ga
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    out = {}
    clk = Clocks(index, clocks_dir)
    clk.start()
    clk.begin()
    for kind, name in ((2, "dp_mix"), (0, "min_max"), (1, "add")):
        iters = 1 << 12
        for _ in range(2):                                  # warm-up launch
            e2ga.e2_probe_int_rate(kind, iters, stream.cuda_stream)
        st, ops, ms = e2ga.e2_probe_int_rate(kind, iters, stream.cuda_stream)
        if st == 0 and ms > 0:                               # ~20 ms per timed launch
            iters = max(1, min(1 << 24, int(iters * 20.0 / ms)))
        best = None
        for _ in range(5):
            st, ops, ms = e2ga.e2_probe_int_rate(kind, iters, stream.cuda_stream)
            if st != 0:
                raise RuntimeError(f"e2_probe_int_rate failed ({st})")
            rate = ops / (ms * 1e-3)
            best = rate if best is None else max(best, rate)
        out[name] = best
    clk.end()
    c = clk.stop() or {}
    mhz = c.get("sm_mhz") or 0.0
    per_clk = {k: (v / (sms * mhz * 1e6) if mhz else None) for k, v in out.items()}
    return {"ops_per_s": out, "ops_per_sm_per_clock": per_clk, "sm_count": sms, "clocks": c}


def measure(torch, eng, prob, seed, steps, warmup, flush, flush_between=True):
    """`warmup` untimed then `steps` timed generations of a device-resident
    search through e2_run_generation (a recorded launch sequence), each timed
    by CUDA events on the engine's stream; the DP kernel's own duration comes
    from the events recorded around its launches, read after every step."""
    stream = eng.stream
    dpx, dpy = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    dpx.record(stream)                     # torch creates the CUDA event at its first record
    dpy.record(stream)
    eng.set_timing_events(dpx, dpy)
    eng.init_population(seed)
    gen = 0
    for _ in range(warmup):                # also records the launch sequence of both population buffers
        gen += 1
        if prob.redraw:
            eng.redraw_congestion(seed, gen)
        eng.run_generation(seed, gen)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    stats, dp_ms = [], []
    launched = eng.stats()["launches"]     # the library's own count of its kernel launches
    torch.cuda.synchronize()
    if not flush_between:
        with torch.cuda.stream(stream):
            flush.fill_(7)
    for i in range(steps):
        if flush_between:
            with torch.cuda.stream(stream):
                flush.fill_(i & 0xFF)
        gen += 1
        a, c = ev[i]
        a.record(stream)
        if prob.redraw:                    # congestion redrawn every generation
            eng.redraw_congestion(seed, gen)
        eng.run_generation(seed, gen)
        c.record(stream)
        if flush_between:
            stats.append(eng.stats())      # synchronises
            dp_ms.append(dpx.elapsed_time(dpy))
    torch.cuda.synchronize()
    if not flush_between:                  # back to back: only the last step's DP events are read
        stats.append(eng.stats())
        dp_ms.append(dpx.elapsed_time(dpy))
    eng.set_timing_events()
    step_ms = [a.elapsed_time(c) for a, c in ev]
    n = len(stats)
    probes = sum(s["dp_probes"] for s in stats) / n
    cells = sum(s["dp_cells"] for s in stats) / n
    return {"gen": gen, "step_ms": step_ms, "t_s": sum(step_ms) / 1e3, "stats": stats,
            "launches": eng.stats()["launches"] - launched,
            "dp_s": sum(dp_ms) / 1e3 / n, "probes": probes, "cells": cells,
            "ops": OPS_PER_PROBE * probes + OPS_PER_CELL * cells,
            "paper": sum(s["paper_candidates"] for s in stats) / n}


def config_line(torch, name, seed, peak_ops, flush, roles):
    """Device-timed line of another workload (own engine, freed afterwards)."""
    prob = W.make_config(name)
    if roles == "search" and prob.K_max <= 20:
        prob = dataclasses.replace(prob, role_search=1)
    from paper_2606_03770_gb300.e2ga import Engine
    eng = Engine(prob)
    gens = max(prob.G, 10)
    back_to_back = prob.G >= 100          # the end-to-end GA: generations per second
    m = measure(torch, eng, prob, seed, gens, 3, flush, flush_between=not back_to_back)
    eng.close()
    del eng
    achieved = m["ops"] / m["dp_s"]
    line = {"workload": workload_label(prob), "generations": gens,
            "genomes_per_s": prob.P * gens / m["t_s"], "ms_per_generation": 1e3 * m["t_s"] / gens,
            "dp_kernel_ms_per_generation": 1e3 * m["dp_s"], "dp_ops_per_s": achieved,
            "dp_frac_of_measured_int_peak": achieved / peak_ops if peak_ops else None,
            "served_replicas": m["stats"][-1]["served"], "replicas": m["stats"][-1]["replicas"],
            "l2": "flushed between generations" if not back_to_back else "not flushed (back-to-back generations)"}
    if back_to_back:
        line["generations_per_s"] = gens / m["t_s"]
    return line


def run_ours(args):
    import torch
    import torch.distributed as dist

    rank, world, local = dist_info()
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    import __graft_entry__ as ge
    ge.build()
    from paper_2606_03770_gb300.e2ga import Engine

    prob = problem(args)
    seed = args.seed + 1000 * rank
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()
    peak = int_peak(torch, stream, args.clocks_dir, local) if rank == 0 else None
    peak_ops = peak["ops_per_s"]["dp_mix"] if peak else None

    eng = Engine(prob)

    def sync_all():
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
            torch.cuda.synchronize()

    # ---- device-resident search: one generation per step
    clocks = Clocks(local, args.clocks_dir)
    clocks.start()
    sync_all()
    clocks.begin()
    m = measure(torch, eng, prob, seed, args.steps, args.warmup, flush)
    sync_all()
    clocks.end()
    clk = clocks.stop()
    t_max = max_over_ranks(m["t_s"], world, "cuda")
    value = replica_throughput(prob.P * args.steps, world, t_max)
    stats = m["stats"]
    gen = m["gen"]

    # ---- roofline of the dominant kernel (DP_Pipe evaluation)
    achieved = m["ops"] / m["dp_s"]
    sm_max = clk["sm_max_mhz"] if clk else 2070.0
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    nominal = sms * INT32_LANES_PER_SM * sm_max * 1e6

    # ---- end to end through the C ABI with pinned host buffers
    e2e = None
    if not args.no_e2e:
        P, M, K = prob.P, prob.M, prob.K_max
        def pinned_population():
            return dict(perm=torch.empty((P, M), dtype=torch.int16).pin_memory(),
                        sizes=torch.empty((P, K), dtype=torch.int16).pin_memory(),
                        nclus=torch.empty(P, dtype=torch.uint8).pin_memory(),
                        roles=torch.empty(P, dtype=torch.int64).pin_memory())
        host = [pinned_population(), pinned_population()]
        hfit = torch.empty((P, 4), dtype=torch.float64).pin_memory()
        eng.get_population(host[0])
        bytes_pop = P * (2 * M + 2 * K + 1 + 8)

        def e2e_step(g):
            # the population in from the host (validated on the device), one
            # generation, its fitness and the next population back to the host:
            # one call, one synchronisation
            if prob.redraw:
                eng.redraw_congestion(seed, g)
            eng.run_generation_io(seed, g, population=host[0], fitness=hfit, next_out=host[1])
            host.reverse()

        for _ in range(args.warmup):
            gen += 1
            e2e_step(gen)
        sync_all()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            gen += 1
            e2e_step(gen)
        sync_all()
        te = max_over_ranks(time.perf_counter() - t0, world, "cuda")
        e2e = {"value": replica_throughput(P * args.steps, world, te), "unit": UNIT,
               "h2d_bytes_per_step": bytes_pop, "d2h_bytes_per_step": bytes_pop + 32 * P + 4,
               "call": "e2_run_generation_io (population in, fitness and next population out)"}
    eng.close()
    del eng

    if rank == 0:
        n = len(stats)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * t_max / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded fleet, links and dense-decoder profile; no paper data)",
            "config": {"workload": workload_label(prob),
                       "l2": "flushed (256 MB write) between timed steps",
                       "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
            "gpu_launches": m["launches"],
            "dp_cells_per_s": m["cells"] * args.steps * world / t_max,
            "paper_candidates_per_s": m["paper"] * args.steps * world / t_max,
            "dp_kernel_ms_per_step": 1e3 * m["dp_s"],
            "served_replicas_per_step": sum(s["served"] for s in stats) / n,
            "prepass_per_step": {"memory_rejected": sum(s["prechecked"] for s in stats) / n,
                                 "latency_rejected": sum(s["tps_pruned"] for s in stats) / n},
            "dp_launches": {"ctas": [stats[-1]["dp_ctas"], stats[-1]["dp_ctas_small"]],
                            "smem_bytes": [stats[-1]["dp_smem"], stats[-1]["dp_smem_small"]],
                            "runs": [sum(s["dp_runs"] - s["dp_runs_small"] for s in stats) / n,
                                     sum(s["dp_runs_small"] for s in stats) / n]},
            "replicas_per_step": sum(s["replicas"] for s in stats) / n,
            "roofline": {"bound": "alu",
                         "kernel": "dp_eval_kernel (DP_Pipe; both launches, timed by events around them)",
                         "achieved": achieved / 1e12, "peak": peak_ops / 1e12 if peak_ops else None,
                         "unit": "Tops/s (int32)", "frac": achieved / peak_ops if peak_ops else None,
                         "traffic": DP_TRAFFIC_BYTES if args.config == WORKLOAD else None,
                         "traffic_source": DP_TRAFFIC_SOURCE,
                         "per_unit": f"{OPS_PER_PROBE} int32 ops per crossover probe + {OPS_PER_CELL} per DP cell "
                                     f"(about five per examined candidate); probes {m['probes']:.4g} and cells "
                                     f"{m['cells']:.4g} per step, the kernel's own tallies",
                         "peak_source": "measured in this run: e2_probe_int_rate kind 2 (min, max, compare, "
                                        "select, add on independent chains at full occupancy), best of 5",
                         "peak_nominal": nominal / 1e12,
                         "frac_of_nominal": achieved / nominal,
                         "nominal_source": f"{sms} SMs x {INT32_LANES_PER_SM} int32 lanes x {sm_max:.0f} MHz"},
            "int_peak_probe": peak,
            "e2e": e2e,
            "clocks": clk,
        }
        if world == 1 and not args.no_configs:
            line["configs"] = {c: config_line(torch, c, seed, peak_ops, flush, args.roles) for c in OTHER_CONFIGS
                               if c != args.config}
        if not args.no_cpu and world == 1:
            line["cpu_baseline"] = cpu_baseline(prob, seed)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def replica_keys(pop, P, K, N):
    """(ordered device tuple, role) of every replica of a population, with the
    size of its DP runs (m x (N - m + 1), 0 when it has more devices than
    blocks and runs none)."""
    keys, work = [], []
    for g in range(P):
        off = 0
        R = int(pop["nclus"][g])
        roles = int(pop["roles"][g])
        perm = pop["perm"][g]
        for c in range(R):
            m = int(pop["sizes"][g][c])
            keys.append((perm[off:off + m].tobytes(), (roles >> c) & 1))
            work.append(m * (N - m + 1) if m <= N else 0)
            off += m
    return keys, work


def run_repeats(args):
    """How often a replica (its ordered devices and role) that the evaluation
    meets was already evaluated: within the same generation, and within the
    last `window` generations (what a per-replica result cache, Sec. 3.4,
    would serve), over a long run of the search, by count and by DP work."""
    import torch
    import __graft_entry__ as ge
    ge.build()
    from paper_2606_03770_gb300.e2ga import Engine
    prob = problem(args)
    eng = Engine(prob)
    eng.init_population(args.seed)
    window, marks = 5, {1, 2, 10, 50, 100, 150, max(prob.G, 2)}
    keep = {g for m in marks for g in range(max(1, m - window), m + 1)}
    hist, rows = {}, []
    for gen in range(1, max(prob.G, 2) + 1):
        if gen in keep:
            pop = eng.get_population()
            hist[gen] = replica_keys(pop, prob.P, prob.K_max, prob.N)
        if gen in marks:
            keys, work = hist[gen]
            seen, within, within_w = set(), 0, 0
            for k, w in zip(keys, work):
                if k in seen:
                    within += 1
                    within_w += w
                seen.add(k)
            past = set()
            for g2 in range(max(1, gen - window), gen):
                past.update(hist[g2][0])
            cache, cache_w = 0, 0
            seen = set()
            for k, w in zip(keys, work):
                if k in seen or k in past:
                    cache += 1
                    cache_w += w
                seen.add(k)
            tw = max(1, sum(work))
            rows.append({"generation": gen, "replicas": len(keys),
                         "repeat_within_generation": within / len(keys),
                         "repeat_within_generation_work": within_w / tw,
                         f"hit_cache_last_{window}_generations": cache / len(keys),
                         f"hit_cache_last_{window}_generations_work": cache_w / tw})
        eng.run_generation(args.seed, gen)
    torch.cuda.synchronize()
    eng.close()
    print(json.dumps({"workload": workload_label(prob), "generations": max(prob.G, 2), "rates": rows}), flush=True)


def main():
    args = parse()
    if args.cpu_only:
        prob = problem(args)
        print(json.dumps({"workload": workload_label(prob), "cpu_baseline": cpu_baseline(prob, args.seed)}),
              flush=True)
    elif args.repeats:
        run_repeats(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
