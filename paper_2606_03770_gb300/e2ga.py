"""Thin Python binding of the e2ga C ABI (include/e2ga.h).

Every ``e2_*`` function here marshals arguments into the shared library and
returns its status; all computation happens in the library's CUDA kernels.
PyTorch provides the device workspace (the library allocates no device
memory) and the CUDA stream.  ``Engine`` bundles the calls of a search.

There is no CPU fallback: if the library has not been built, ``load()``
raises.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libe2ga.so")
_lib = None

E2_OK, E2_EINVAL, E2_ENOMEM, E2_ECUDA, E2_EDEVICE, E2_ESTATE = 0, 1, 2, 3, 5, 6


class e2_devices(C.Structure):
    _fields_ = [("M", C.c_int32), ("rate", C.c_void_p), ("bw", C.c_void_p), ("mem", C.c_void_p),
                ("rate_cpu", C.c_void_p), ("bw_cpu", C.c_void_p), ("mem_cpu", C.c_void_p)]


class e2_links(C.Structure):
    _fields_ = [("bw", C.c_void_p), ("cong", C.c_void_p), ("cong_lo", C.c_double), ("cong_hi", C.c_double)]


class e2_layer_profile(C.Structure):
    _fields_ = [("N", C.c_int32), ("b_max", C.c_int32), ("blk_flops", C.c_void_p), ("blk_bytes", C.c_void_p),
                ("blk_mem", C.c_void_p), ("head_flops", C.c_void_p), ("head_bytes", C.c_void_p),
                ("head_mem", C.c_void_p), ("act_bytes", C.c_void_p), ("NP", C.c_uint64), ("ND", C.c_uint64),
                ("PF", C.c_void_p), ("PB", C.c_void_p), ("PM", C.c_void_p)]


class e2_params(C.Structure):
    _fields_ = [("P", C.c_int32), ("Q", C.c_int32), ("K_max", C.c_int32), ("tournament", C.c_int32),
                ("min_tps", C.c_double), ("t_a", C.c_double), ("p_cx", C.c_double), ("p_mut", C.c_double),
                ("p_swap", C.c_double), ("p_regroup", C.c_double), ("p_regroup_all", C.c_double),
                ("role_search", C.c_int32), ("objective", C.c_int32)]


class e2_genomes(C.Structure):
    _fields_ = [("perm", C.c_void_p), ("sizes", C.c_void_p), ("nclus", C.c_void_p), ("roles", C.c_void_p)]


class e2_partitions(C.Structure):
    _fields_ = [("layers", C.c_void_p), ("master", C.c_void_p), ("bsel", C.c_void_p), ("T", C.c_void_p),
                ("lambda_", C.c_void_p), ("gpu_layers", C.c_void_p)]


class e2_stats(C.Structure):
    _fields_ = [(n, C.c_uint64) for n in ("genomes", "replicas", "dp_runs", "dp_cells", "dp_probes",
                                         "paper_candidates", "prechecked", "served", "tps_pruned",
                                         "dp_runs_small", "dp_launches", "dp_ctas", "dp_smem", "dp_ctas_small",
                                         "dp_smem_small", "launches", "role_search_capped", "device_errors",
                                         "dp_runs_per_cta_small")]


# name -> (restype, argtypes); the exported surface of include/e2ga.h
SIGNATURES = {
    "e2_workspace_bytes": (C.c_size_t, [C.c_int32] * 6),
    "e2_workspace_bytes_ex": (C.c_size_t, [C.c_int32] * 6 + [C.c_uint32]),
    "e2_create": (C.c_int, [C.c_void_p] * 5 + [C.c_size_t, C.c_void_p, C.c_void_p]),
    "e2_destroy": (C.c_int, [C.c_void_p]),
    "e2_set_population": (C.c_int, [C.c_void_p, C.c_void_p]),
    "e2_get_population": (C.c_int, [C.c_void_p, C.c_void_p]),
    "e2_init_population": (C.c_int, [C.c_void_p, C.c_uint64]),
    "e2_eval_population": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "e2_ga_step": (C.c_int, [C.c_void_p, C.c_uint64, C.c_uint32]),
    "e2_redraw_congestion": (C.c_int, [C.c_void_p, C.c_uint64, C.c_uint32]),
    "e2_get_congestion": (C.c_int, [C.c_void_p, C.c_void_p]),
    "e2_get_elites": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "e2_get_stats": (C.c_int, [C.c_void_p, C.c_void_p]),
    "e2_set_timing_events": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "e2_run_generation": (C.c_int, [C.c_void_p, C.c_uint64, C.c_uint32]),
    "e2_run_generation_io": (C.c_int, [C.c_void_p, C.c_void_p, C.c_uint64, C.c_uint32, C.c_void_p,
                                       C.c_void_p]),
    "e2_get_results": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "e2_select_elites_noalloc": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_int32,
                                            C.c_int32, C.c_void_p, C.c_void_p]),
    "e2_probe_int_rate": (C.c_int, [C.c_int32, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p]),
    "e2_strerror": (C.c_char_p, [C.c_int]),
    "e2_last_error": (C.c_char_p, [C.c_void_p]),
}


def load(path: str = LIB_PATH):
    """Load the compiled library; raises if it is missing (no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise RuntimeError(f"e2ga CUDA library not built ({path}); run __graft_entry__.build()")
        lib = C.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(lib, name)
            f.restype, f.argtypes = res, args
        _lib = lib
    return _lib


class E2Error(RuntimeError):
    def __init__(self, status, where, detail=""):
        self.status = status
        msg = load().e2_strerror(status).decode()
        super().__init__(f"{where}: {msg} ({status}){': ' + detail if detail else ''}")


# ---- same-named thin wrappers ------------------------------------------------
E2_WS_LAYERED = 1


def e2_workspace_bytes(M, N, b_max, P, Q, K_max):
    return load().e2_workspace_bytes(M, N, b_max, P, Q, K_max)


def e2_workspace_bytes_ex(M, N, b_max, P, Q, K_max, flags):
    return load().e2_workspace_bytes_ex(M, N, b_max, P, Q, K_max, flags)


def e2_create(devs, links, prof, prm, workspace_ptr, workspace_bytes, stream_ptr):
    ctx = C.c_void_p()
    st = load().e2_create(C.byref(devs), C.byref(links), C.byref(prof), C.byref(prm), workspace_ptr,
                          workspace_bytes, stream_ptr, C.byref(ctx))
    return st, ctx


def e2_destroy(ctx):
    return load().e2_destroy(ctx)


def e2_set_population(ctx, g):
    return load().e2_set_population(ctx, C.byref(g))


def e2_get_population(ctx, g):
    return load().e2_get_population(ctx, C.byref(g))


def e2_init_population(ctx, seed):
    return load().e2_init_population(ctx, seed)


def e2_eval_population(ctx, genomes, fitness_ptr, parts):
    return load().e2_eval_population(ctx, C.byref(genomes) if genomes is not None else None, fitness_ptr,
                                     C.byref(parts) if parts is not None else None)


def e2_ga_step(ctx, seed, generation):
    return load().e2_ga_step(ctx, seed, generation)


def e2_redraw_congestion(ctx, seed, generation):
    return load().e2_redraw_congestion(ctx, seed, generation)


def e2_get_congestion(ctx, ptr):
    return load().e2_get_congestion(ctx, ptr)


def e2_get_elites(ctx, idx_ptr, fit_ptr):
    return load().e2_get_elites(ctx, idx_ptr, fit_ptr)


def e2_get_stats(ctx, stats):
    return load().e2_get_stats(ctx, C.byref(stats))


def e2_get_results(ctx, fitness_ptr, parts):
    return load().e2_get_results(ctx, fitness_ptr, C.byref(parts) if parts is not None else None)


def e2_run_generation(ctx, seed, generation):
    return load().e2_run_generation(ctx, seed, generation)


def e2_run_generation_io(ctx, population, seed, generation, fitness_ptr, next_out):
    return load().e2_run_generation_io(ctx, C.byref(population) if population is not None else None, seed,
                                       generation, fitness_ptr, C.byref(next_out) if next_out is not None else None)


def e2_set_timing_events(ctx, start_ptr, stop_ptr):
    return load().e2_set_timing_events(ctx, start_ptr, stop_ptr)


def e2_select_elites_noalloc(genomes, fitness_ptr, P, M, K_max, Q, elite_ptr, stream_ptr):
    return load().e2_select_elites_noalloc(C.byref(genomes), fitness_ptr, P, M, K_max, Q, elite_ptr, stream_ptr)


def e2_probe_int_rate(kind, iters, stream_ptr):
    """(status, operations executed, milliseconds) of one probe launch."""
    ops, ms = C.c_double(), C.c_float()
    st = load().e2_probe_int_rate(kind, iters, stream_ptr, C.byref(ops), C.byref(ms))
    return st, ops.value, ms.value


def e2_strerror(status):
    return load().e2_strerror(status).decode()


def e2_last_error(ctx):
    return load().e2_last_error(ctx).decode()


# ---- convenience --------------------------------------------------------------
def _ptr(x):
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        assert x.flags["C_CONTIGUOUS"]
        return x.ctypes.data
    return x.data_ptr()   # torch tensor (host or device)


def _check(st, where, ctx=None):
    if st != E2_OK:
        raise E2Error(st, where, e2_last_error(ctx))


class Engine:
    """One search context on the current CUDA device (see include/e2ga.h)."""

    def __init__(self, prob, stream=None):
        import torch
        self.torch = torch
        self.prob = prob
        self.M, self.N, self.P, self.K = prob.M, prob.N, prob.P, prob.K_max
        self.Q, self.b_max = prob.Q, prob.b_max
        f64 = lambda x: np.ascontiguousarray(x, dtype=np.float64)
        u64 = lambda x: np.ascontiguousarray(x, dtype=np.uint64)
        self._host = dict(rate=f64(prob.rate), bw=f64(prob.bw), mem=u64(prob.mem), lbw=f64(prob.link_bw),
                          cong=f64(prob.cong), blk_flops=u64(prob.blk_flops), blk_bytes=u64(prob.blk_bytes),
                          blk_mem=u64(prob.blk_mem), head_flops=u64(prob.head_flops),
                          head_bytes=u64(prob.head_bytes), head_mem=u64(prob.head_mem),
                          act_bytes=u64(prob.act_bytes))
        if getattr(prob, "mem_cpu", None) is not None:
            self._host.update(rate_cpu=f64(prob.rate_cpu), bw_cpu=f64(prob.bw_cpu), mem_cpu=u64(prob.mem_cpu))
        h = self._host
        self.devs = e2_devices(self.M, _ptr(h["rate"]), _ptr(h["bw"]), _ptr(h["mem"]), _ptr(h.get("rate_cpu")),
                               _ptr(h.get("bw_cpu")), _ptr(h.get("mem_cpu")))
        self.links = e2_links(_ptr(h["lbw"]), _ptr(h["cong"]), prob.cong_lo, prob.cong_hi)
        layered = getattr(prob, "PF", None) is not None
        if layered:
            self._host.update(PF=u64(prob.PF), PB=u64(prob.PB), PM=u64(prob.PM))
        self.profile = e2_layer_profile(self.N, self.b_max, *[_ptr(h[k]) for k in (
            "blk_flops", "blk_bytes", "blk_mem", "head_flops", "head_bytes", "head_mem", "act_bytes")],
            prob.NP, prob.ND, *[_ptr(h.get(k)) for k in ("PF", "PB", "PM")])
        pk = prob.p_kind
        self.params = e2_params(self.P, self.Q, self.K, prob.tournament, prob.min_tps, prob.t_a, prob.p_cx,
                                prob.p_mut, pk[0], pk[1], pk[2], int(getattr(prob, "role_search", 0)),
                                int(getattr(prob, "objective", 0)))
        self.ws_bytes = e2_workspace_bytes_ex(self.M, self.N, self.b_max, self.P, self.Q, self.K,
                                              E2_WS_LAYERED if layered else 0)
        if self.ws_bytes == 0:
            raise E2Error(E2_EINVAL, "e2_workspace_bytes")
        self.workspace = torch.empty(self.ws_bytes, dtype=torch.uint8, device="cuda")
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        st, ctx = e2_create(self.devs, self.links, self.profile, self.params, self.workspace.data_ptr(),
                            self.ws_bytes, self.stream.cuda_stream)
        _check(st, "e2_create", None)
        self.ctx = ctx
        dev = torch.device("cuda")
        self.fitness = torch.empty((self.P, 4), dtype=torch.float64, device=dev)
        self.layers = torch.empty((self.P, self.M), dtype=torch.int16, device=dev)
        self.master = torch.empty((self.P, self.K), dtype=torch.int16, device=dev)
        self.bsel = torch.empty((self.P, self.K), dtype=torch.int16, device=dev)
        self.T = torch.empty((self.P, self.K), dtype=torch.float64, device=dev)
        self.L = torch.empty((self.P, self.K), dtype=torch.float64, device=dev)
        self.gpu_layers = torch.empty((self.P, self.M), dtype=torch.int16, device=dev)

    # -- population ------------------------------------------------------------
    def genome_struct(self, g):
        return e2_genomes(_ptr(g["perm"]), _ptr(g["sizes"]), _ptr(g["nclus"]), _ptr(g["roles"]))

    def set_population(self, g):
        _check(e2_set_population(self.ctx, self.genome_struct(g)), "e2_set_population", self.ctx)

    def get_population(self, out=None):
        if out is None:
            out = dict(perm=np.zeros((self.P, self.M), np.uint16), sizes=np.zeros((self.P, self.K), np.uint16),
                       nclus=np.zeros(self.P, np.uint8), roles=np.zeros(self.P, np.uint64))
        _check(e2_get_population(self.ctx, self.genome_struct(out)), "e2_get_population", self.ctx)
        return out

    def init_population(self, seed):
        _check(e2_init_population(self.ctx, seed), "e2_init_population", self.ctx)

    # -- evaluation and search -------------------------------------------------
    def eval(self, genomes=None, fitness=None, parts=True):
        """Evaluate; results land in the engine's device tensors (or in the
        given fitness buffer / host arrays)."""
        gs = self.genome_struct(genomes) if genomes is not None else None
        fit = self.fitness if fitness is None else fitness
        ps = None
        if parts is True:
            ps = e2_partitions(_ptr(self.layers), _ptr(self.master), _ptr(self.bsel), _ptr(self.T), _ptr(self.L),
                               _ptr(self.gpu_layers))
        elif isinstance(parts, dict):
            ps = e2_partitions(*[_ptr(parts.get(k)) for k in ("layers", "master", "bsel", "T", "L", "gpu_layers")])
        _check(e2_eval_population(self.ctx, gs, _ptr(fit), ps), "e2_eval_population", self.ctx)
        return fit

    def results(self):
        """The most recent evaluation's results, as numpy arrays."""
        ps = e2_partitions(_ptr(self.layers), _ptr(self.master), _ptr(self.bsel), _ptr(self.T), _ptr(self.L),
                           _ptr(self.gpu_layers))
        _check(e2_get_results(self.ctx, _ptr(self.fitness), ps), "e2_get_results", self.ctx)
        self.torch.cuda.synchronize()
        return dict(fitness=self.fitness.cpu().numpy(), layers=self.layers.cpu().numpy(),
                    master=self.master.cpu().numpy(), bsel=self.bsel.cpu().numpy(), T=self.T.cpu().numpy(),
                    L=self.L.cpu().numpy(), gpu_layers=self.gpu_layers.cpu().numpy())

    def ga_step(self, seed, generation):
        _check(e2_ga_step(self.ctx, seed, generation), "e2_ga_step", self.ctx)

    def run_generation(self, seed, generation):
        """Evaluation, elites and next population in one recorded launch."""
        _check(e2_run_generation(self.ctx, seed, generation), "e2_run_generation", self.ctx)

    def run_generation_io(self, seed, generation, population=None, fitness=None, next_out=None):
        """One generation with the host in the loop: optionally upload a
        population, run the generation, copy the fitness and the next
        population out (any of them host or device arrays); one
        synchronisation."""
        pin = self.genome_struct(population) if population is not None else None
        pout = self.genome_struct(next_out) if next_out is not None else None
        _check(e2_run_generation_io(self.ctx, pin, seed, generation, _ptr(fitness), pout),
               "e2_run_generation_io", self.ctx)

    def redraw_congestion(self, seed, generation):
        _check(e2_redraw_congestion(self.ctx, seed, generation), "e2_redraw_congestion", self.ctx)

    def congestion(self):
        out = np.zeros((self.M, self.M), np.float64)
        _check(e2_get_congestion(self.ctx, _ptr(out)), "e2_get_congestion", self.ctx)
        return out

    def elites(self):
        idx = np.zeros(max(self.Q, 1), np.int32)
        fit = np.zeros((max(self.Q, 1), 4), np.float64)
        _check(e2_get_elites(self.ctx, _ptr(idx), _ptr(fit)), "e2_get_elites", self.ctx)
        return idx[:self.Q], fit[:self.Q]

    def set_timing_events(self, start=None, stop=None):
        """Record two torch.cuda.Events around the DP kernel of later evaluations."""
        sp = start.cuda_event if start is not None else None
        ep = stop.cuda_event if stop is not None else None
        _check(e2_set_timing_events(self.ctx, sp, ep), "e2_set_timing_events", self.ctx)

    def stats(self):
        s = e2_stats()
        _check(e2_get_stats(self.ctx, s), "e2_get_stats", self.ctx)
        return {n: int(getattr(s, n)) for n, _ in e2_stats._fields_}

    def close(self):
        if getattr(self, "ctx", None):
            e2_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
