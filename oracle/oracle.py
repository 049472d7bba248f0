"""ctypes binding for the plain C oracle (test infrastructure only).

Only the tests, the smoke check and the benchmark's CPU-baseline leg import
this module.  The CUDA library never does, and this module imports nothing
from the CUDA side: it takes the same seeded inputs as plain numpy arrays.

``build()`` compiles ``e2_oracle.c`` with ``-O2 -ffp-contract=off`` (no fused
multiply-add, so every float64 operation rounds once, as on the device) and
OpenMP for the all-cores CPU baseline.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.environ.get("E2_ORACLE_SRC", os.path.join(_HERE, "e2_oracle.c"))
_OUT = os.environ.get("E2_ORACLE_LIB", os.path.join(_HERE, "_build", "libe2oracle.so"))
_lib = None

PURPOSE = dict(INIT_PERM=0, INIT_GROUP=1, INIT_ROLES=2, SELECT=3, CROSS=4, MUTATE=5,
               MUT_PERM=6, MUT_GROUP=7, MUT_ROLES=8, CONG=9)


def build(force: bool = False) -> str:
    os.makedirs(os.path.dirname(_OUT), exist_ok=True)
    if force or not os.path.exists(_OUT) or os.path.getmtime(_OUT) < os.path.getmtime(_SRC):
        cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-fopenmp",
               _SRC, "-o", _OUT + ".tmp", "-lm"]
        subprocess.check_call(cmd)
        os.replace(_OUT + ".tmp", _OUT)
    return _OUT


class _Problem(C.Structure):
    _fields_ = [("M", C.c_int), ("N", C.c_int), ("V", C.c_int),
                ("rate", C.c_void_p), ("bw", C.c_void_p), ("mem", C.c_void_p),
                ("link_bw", C.c_void_p), ("cong", C.c_void_p),
                ("blk_flops", C.c_void_p), ("blk_bytes", C.c_void_p), ("blk_mem", C.c_void_p),
                ("head_flops", C.c_void_p), ("head_bytes", C.c_void_p), ("head_mem", C.c_void_p),
                ("act_bytes", C.c_void_p), ("NP", C.c_uint64), ("ND", C.c_uint64),
                ("min_tps", C.c_double), ("t_a", C.c_double), ("role_search", C.c_int),
                ("objective", C.c_int), ("rate_cpu", C.c_void_p), ("bw_cpu", C.c_void_p),
                ("mem_cpu", C.c_void_p), ("PF", C.c_void_p), ("PB", C.c_void_p), ("PM", C.c_void_p)]


class _GA(C.Structure):
    _fields_ = [("P", C.c_int), ("M", C.c_int), ("K", C.c_int), ("Q", C.c_int),
                ("tournament", C.c_int), ("p_cx", C.c_double), ("p_mut", C.c_double),
                ("p_swap", C.c_double), ("p_regroup", C.c_double), ("p_regroup_all", C.c_double)]


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(build())
        _lib.orc_stage_cost.restype = C.c_double
        _lib.orc_stage_cost.argtypes = [C.c_void_p, C.c_int, C.c_int, C.c_int, C.c_int]
        _lib.orc_stage_cost_at.restype = C.c_double
        _lib.orc_stage_cost_at.argtypes = [C.c_void_p, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int]
        _lib.orc_gpu_blocks.restype = C.c_int
        _lib.orc_gpu_blocks.argtypes = [C.c_void_p, C.c_int, C.c_int, C.c_int, C.c_int]
        _lib.orc_link_cost.restype = C.c_double
        _lib.orc_link_cost.argtypes = [C.c_void_p, C.c_int, C.c_int, C.c_int]
        _lib.orc_dp_pipe.restype = C.c_int
        _lib.orc_dp_pipe.argtypes = [C.c_void_p, C.c_int, C.c_void_p, C.c_int, C.c_void_p,
                                     C.c_void_p, C.c_void_p, C.c_void_p]
        _lib.orc_latency.restype = C.c_double
        _lib.orc_latency.argtypes = [C.c_void_p, C.c_int, C.c_void_p, C.c_int, C.c_int, C.c_void_p]
        _lib.orc_eval_cluster.restype = C.c_int
        _lib.orc_eval_cluster.argtypes = [C.c_void_p, C.c_void_p, C.c_int, C.c_int, C.c_void_p,
                                          C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]
        _lib.orc_score.restype = None
        _lib.orc_score.argtypes = [C.c_void_p, C.c_int, C.c_uint64, C.c_void_p, C.c_void_p, C.c_void_p,
                                   C.c_void_p]
        _lib.orc_splitwise_prefill_count.restype = C.c_int
        _lib.orc_splitwise_prefill_count.argtypes = [C.c_uint64, C.c_uint64, C.c_int]
        _lib.orc_eval_population.restype = None
        _lib.orc_eval_population.argtypes = [C.c_void_p, C.c_int, C.c_int] + [C.c_void_p] * 11 + [C.c_int,
                                                                                                   C.c_void_p,
                                                                                                   C.c_void_p]
        _lib.orc_philox4x32_10.restype = None
        _lib.orc_philox4x32_10.argtypes = [C.c_void_p, C.c_void_p, C.c_void_p]
        _lib.orc_word.restype = C.c_uint32
        _lib.orc_word.argtypes = [C.c_uint64, C.c_uint32, C.c_uint32, C.c_uint32, C.c_uint32]
        _lib.orc_threshold.restype = C.c_uint64
        _lib.orc_threshold.argtypes = [C.c_double]
        _lib.orc_init_population.restype = None
        _lib.orc_init_population.argtypes = [C.c_void_p, C.c_uint64] + [C.c_void_p] * 4
        _lib.orc_elites.restype = None
        _lib.orc_elites.argtypes = [C.c_void_p] + [C.c_void_p] * 6
        _lib.orc_ga_step.restype = None
        _lib.orc_ga_step.argtypes = [C.c_void_p, C.c_uint64, C.c_uint32] + [C.c_void_p] * 10
        _lib.orc_redraw_congestion.restype = None
        _lib.orc_redraw_congestion.argtypes = [C.c_int, C.c_uint64, C.c_uint32, C.c_double,
                                               C.c_double, C.c_void_p]
        _lib.orc_num_threads.restype = C.c_int
        _lib.orc_repair.restype = None
        _lib.orc_repair.argtypes = [C.c_void_p, C.c_int, C.c_void_p]
    return _lib


def _p(a):
    return a.ctypes.data_as(C.c_void_p)


class OracleProblem:
    """Keeps the numpy arrays alive for as long as the C struct points at them."""

    def __init__(self, prob, cong=None):
        self.prob = prob
        f64 = lambda x: np.ascontiguousarray(x, dtype=np.float64)
        u64 = lambda x: np.ascontiguousarray(x, dtype=np.uint64)
        self.arrays = dict(rate=f64(prob.rate), bw=f64(prob.bw), mem=u64(prob.mem),
                           link_bw=f64(prob.link_bw), cong=f64(prob.cong if cong is None else cong),
                           blk_flops=u64(prob.blk_flops), blk_bytes=u64(prob.blk_bytes),
                           blk_mem=u64(prob.blk_mem), head_flops=u64(prob.head_flops),
                           head_bytes=u64(prob.head_bytes), head_mem=u64(prob.head_mem),
                           act_bytes=u64(prob.act_bytes))
        off = getattr(prob, "mem_cpu", None) is not None
        if off:
            self.arrays.update(rate_cpu=f64(prob.rate_cpu), bw_cpu=f64(prob.bw_cpu), mem_cpu=u64(prob.mem_cpu))
        layered = getattr(prob, "PF", None) is not None
        if layered:
            self.arrays.update(PF=u64(prob.PF), PB=u64(prob.PB), PM=u64(prob.PM))
        a = self.arrays
        self.s = _Problem(prob.M, prob.N, prob.V, *[_p(a[k]) for k in
                          ("rate", "bw", "mem", "link_bw", "cong", "blk_flops", "blk_bytes",
                           "blk_mem", "head_flops", "head_bytes", "head_mem", "act_bytes")],
                          prob.NP, prob.ND, prob.min_tps, prob.t_a, int(getattr(prob, "role_search", 0)),
                          int(getattr(prob, "objective", 0)),
                          *([_p(a[k]) for k in ("rate_cpu", "bw_cpu", "mem_cpu")] if off else [None] * 3),
                          *([_p(a[k]) for k in ("PF", "PB", "PM")] if layered else [None] * 3))

    def set_cong(self, cong):
        self.arrays["cong"] = np.ascontiguousarray(cong, dtype=np.float64)
        self.s.cong = _p(self.arrays["cong"])

    @property
    def ref(self):
        return C.byref(self.s)

    def stage_cost(self, v, d, n, master):
        return lib().orc_stage_cost(self.ref, v, d, n, int(master))

    def stage_cost_at(self, v, d, j, n, master):
        return lib().orc_stage_cost_at(self.ref, v, d, j, n, int(master))

    def gpu_blocks(self, v, d, n, master):
        return lib().orc_gpu_blocks(self.ref, v, d, n, int(master))

    def link_cost(self, v, a, b):
        return lib().orc_link_cost(self.ref, v, a, b)

    def dp_pipe(self, v, devs):
        devs = np.ascontiguousarray(devs, dtype=np.uint16)
        m = len(devs)
        V = C.c_double()
        mu = C.c_int()
        layers = np.zeros(max(m, 1), np.int16)
        cand = C.c_uint64(0)
        ok = lib().orc_dp_pipe(self.ref, v, _p(devs), m, C.byref(V), C.byref(mu), _p(layers), C.byref(cand))
        return dict(ok=bool(ok), V=V.value, mu=mu.value, layers=layers[:m].copy(), cand=cand.value)

    def latency(self, v, devs, mu, layers):
        devs = np.ascontiguousarray(devs, dtype=np.uint16)
        layers = np.ascontiguousarray(layers, dtype=np.int16)
        return lib().orc_latency(self.ref, v, _p(devs), len(devs), mu, _p(layers))

    def eval_cluster(self, devs, decode):
        devs = np.ascontiguousarray(devs, dtype=np.uint16)
        m = len(devs)
        T, L = C.c_double(), C.c_double()
        mu, b = C.c_int(), C.c_int()
        layers = np.zeros(max(m, 1), np.int16)
        ok = lib().orc_eval_cluster(self.ref, _p(devs), m, int(decode), C.byref(T), C.byref(L),
                                    C.byref(mu), C.byref(b), _p(layers), None)
        return dict(ok=bool(ok), T=T.value, L=L.value, mu=mu.value, b=b.value, layers=layers[:m].copy())

    def score(self, roles, T, bsel, L=None):
        T = np.ascontiguousarray(T, dtype=np.float64)
        L = np.ascontiguousarray(np.zeros(len(T)) if L is None else L, dtype=np.float64)
        bsel = np.ascontiguousarray(bsel, dtype=np.int16)
        fit = np.zeros(4, np.float64)
        lib().orc_score(self.ref, len(T), int(roles), _p(T), _p(L), _p(bsel), _p(fit))
        return fit

    def eval_population(self, genomes, K, nthreads=1):
        perm = np.ascontiguousarray(genomes["perm"], dtype=np.uint16)
        sizes = np.ascontiguousarray(genomes["sizes"], dtype=np.uint16)
        nclus = np.ascontiguousarray(genomes["nclus"], dtype=np.uint8)
        roles = np.ascontiguousarray(genomes["roles"], dtype=np.uint64)
        P, M = perm.shape
        out = dict(fitness=np.zeros((P, 4), np.float64), layers=np.zeros((P, M), np.int16),
                   master=np.zeros((P, K), np.int16), bsel=np.zeros((P, K), np.int16),
                   T=np.zeros((P, K), np.float64), L=np.zeros((P, K), np.float64),
                   roles=np.zeros(P, np.uint64))
        cand, capped = C.c_uint64(0), C.c_uint64(0)
        lib().orc_eval_population(self.ref, P, K, _p(perm), _p(sizes), _p(nclus), _p(roles),
                                  _p(out["fitness"]), _p(out["layers"]), _p(out["master"]),
                                  _p(out["bsel"]), _p(out["T"]), _p(out["L"]), C.byref(cand),
                                  int(nthreads), _p(out["roles"]), C.byref(capped))
        out["cand"] = cand.value
        out["capped"] = capped.value
        return out


def _ga_struct(P, M, K, Q, tournament, p_cx, p_mut, p_kind):
    return _GA(P, M, K, Q, tournament, p_cx, p_mut, p_kind[0], p_kind[1], p_kind[2])


def ga_of(prob):
    return _ga_struct(prob.P, prob.M, prob.K_max, prob.Q, prob.tournament, prob.p_cx, prob.p_mut,
                      prob.p_kind)


def empty_genomes(P, M, K):
    return dict(perm=np.zeros((P, M), np.uint16), sizes=np.zeros((P, K), np.uint16),
                nclus=np.zeros(P, np.uint8), roles=np.zeros(P, np.uint64))


def init_population(ga, seed):
    g = empty_genomes(ga.P, ga.M, ga.K)
    lib().orc_init_population(C.byref(ga), seed, _p(g["perm"]), _p(g["sizes"]), _p(g["nclus"]),
                              _p(g["roles"]))
    return g


def elites(ga, genomes, fitness):
    idx = np.zeros(max(ga.Q, 1), np.int32)
    fit = np.ascontiguousarray(fitness, dtype=np.float64)
    lib().orc_elites(C.byref(ga), _p(genomes["perm"]), _p(genomes["sizes"]), _p(genomes["nclus"]),
                     _p(genomes["roles"]), _p(fit), _p(idx))
    return idx[:ga.Q].copy()


def ga_step(ga, seed, gen, genomes, fitness, elite_idx):
    nxt = empty_genomes(ga.P, ga.M, ga.K)
    fit = np.ascontiguousarray(fitness, dtype=np.float64)
    eidx = np.ascontiguousarray(elite_idx if len(elite_idx) else np.zeros(1, np.int32), dtype=np.int32)
    lib().orc_ga_step(C.byref(ga), seed, gen, _p(genomes["perm"]), _p(genomes["sizes"]),
                      _p(genomes["nclus"]), _p(genomes["roles"]), _p(fit), _p(eidx),
                      _p(nxt["perm"]), _p(nxt["sizes"]), _p(nxt["nclus"]), _p(nxt["roles"]))
    return nxt


def redraw_congestion(M, seed, gen, lo, hi):
    cong = np.zeros((M, M), np.float64)
    lib().orc_redraw_congestion(M, seed, gen, lo, hi, _p(cong))
    return cong


def philox(ctr, key):
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, np.uint32)
    lib().orc_philox4x32_10(_p(c), _p(k), _p(out))
    return out


def word(seed, gen, slot, purpose, t):
    return lib().orc_word(seed, gen, slot, purpose, t)


def threshold(p):
    return lib().orc_threshold(p)


def repair(perm):
    cp = np.ascontiguousarray(perm, dtype=np.uint16).copy()
    seen = np.zeros(len(cp), np.uint8)
    lib().orc_repair(_p(cp), len(cp), _p(seen))
    return cp


def splitwise_prefill_count(NP, ND, R):
    return lib().orc_splitwise_prefill_count(NP, ND, R)


def num_threads():
    return lib().orc_num_threads()
