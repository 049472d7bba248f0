"""Parity of per-layer profiles (blocks of several types, Sec. 3.1) with the
oracle, through the C ABI.

Models whose blocks alternate sliding-window and full attention (or end in
a run of full-attention blocks), given as per-variant prefix sums PF, PB,
PM: every stage then costs what its own blocks cost, and these contexts run
the plain-scan DP (every split of every cell, the masters factored through
prefix and suffix tables).  Fitness, partitions, T and Lambda bit-exact,
with role bits, the role search and the adapted-SplitWise rule, and over
generations; plus the uniform-sum case against the identical-block kernel
and the inputs e2_create refuses.
"""
import ctypes as C
import dataclasses

import numpy as np
import pytest

from oracle import oracle as O
from paper_2606_03770_gb300 import workloads as W

from test_parity_gpu import _edge_problem, assert_eval_equal, assert_genomes_equal, engine, take

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()


CASES = [("c1_tiny", 64, "alternate", 0), ("c2", 1024, "alternate", 0), ("c2", 512, "tail", 0),
         ("c2", 256, "alternate", 1), ("c2", 256, "tail", 2), ("c3", 256, "alternate", 0)]


@pytest.mark.parametrize("name,P,layered,role_search", CASES)
def test_layered_parity_full_population(name, P, layered, role_search):
    prob = dataclasses.replace(W.make_config(name, P=P, layered=layered), role_search=role_search)
    eng = engine(prob)
    g = W.random_genomes(prob.M, prob.K_max, P, seed=31)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    assert np.array_equal(eng.get_population()["roles"], ora["roles"])
    st = eng.stats()                                      # raises on a device-side check
    assert st["paper_candidates"] == ora["cand"] and st["device_errors"] == 0
    assert st["served"] == int((ora["bsel"] >= 0).sum()) > 0
    eng.close()


def test_layered_tie_heavy_small_integers():
    """Small-integer per-layer work (heavy and light blocks, many exact ties)
    on tight memories: the smallest-split and smallest-master rules."""
    from test_oracle_pins import _layered
    rng = np.random.default_rng(91)
    M, N, K, P = 24, 12, 6, 48
    prob = _layered(_edge_problem(rng, M, N, P, K, integer=True, Q=2, min_tps=0.05), rng, integer=True)
    g = W.random_genomes(M, K, P, seed=12)
    eng = engine(prob)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, K, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    assert np.isfinite(ora["T"]).sum() > 20
    eng.close()


def test_layered_full_size_sampled():
    prob = W.make_config("c5", layered="alternate")
    eng = engine(prob)
    eng.init_population(55)
    g = eng.get_population()
    eng.eval()
    gpu = eng.results()
    idx = np.sort(np.random.default_rng(3).choice(prob.P, 96, replace=False))
    ora = O.OracleProblem(prob).eval_population(take(g, idx), prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora, rows=idx)
    eng.close()


def test_uniform_sums_equal_the_identical_block_kernel():
    """Prefix sums of identical blocks through the plain-scan path give what
    the identical-block kernel gives (and what the oracle gives)."""
    prob = W.make_config("c2", P=512)
    ramp = np.arange(prob.N + 1, dtype=np.uint64)[None, :]
    lay = dataclasses.replace(prob, PF=prob.blk_flops[:, None] * ramp, PB=prob.blk_bytes[:, None] * ramp,
                              PM=prob.blk_mem[:, None] * ramp)
    g = W.random_genomes(prob.M, prob.K_max, prob.P, seed=8)
    a, b = engine(prob), engine(lay)
    a.eval(g)
    b.eval(g)
    ra, rb = a.results(), b.results()
    for k in ("fitness", "layers", "master", "bsel", "T", "L"):
        assert np.array_equal(ra[k], rb[k]), k
    a.close()
    b.close()


def test_layered_generations():
    prob = W.make_config("c2", P=256, layered="alternate")
    ga = O.ga_of(prob)
    op = O.OracleProblem(prob)
    eng = engine(prob)
    eng.init_population(19)
    pop = O.init_population(ga, 19)
    for gen in range(1, 4):
        ora = op.eval_population(pop, prob.K_max, nthreads=O.num_threads())
        if gen % 2:
            eng.run_generation(19, gen)
        else:
            eng.eval(parts=False)
            eng.ga_step(19, gen)
        assert np.array_equal(eng.results()["fitness"], ora["fitness"]), gen
        pop = O.ga_step(ga, 19, gen, pop, ora["fitness"], O.elites(ga, pop, ora["fitness"]))
        assert_genomes_equal(eng.get_population(), pop)
    eng.close()


def test_layered_inputs_refused():
    """Per-layer sums with GPU-CPU offload, too many blocks, decreasing sums, or
    a workspace sized without the per-layer table: statuses, no launch."""
    from paper_2606_03770_gb300 import e2ga
    lib = e2ga.load()
    base = W.make_config("c1_tiny", layered="alternate")
    host = W.make_config("c1_tiny", layered="alternate", offload=True)
    bad = base.PF.copy()
    bad[0, 5] = bad[0, 4] - np.uint64(1)
    for prob, why in ((host, "offload"), (dataclasses.replace(base, PF=bad), "decreasing")):
        with pytest.raises(e2ga.E2Error) as err:
            e2ga.Engine(prob)
        assert err.value.status == e2ga.E2_EINVAL, why
    assert lib.e2_workspace_bytes_ex(8, 181, 8, 64, 2, 2, e2ga.E2_WS_LAYERED) == 0
    assert lib.e2_workspace_bytes_ex(8, 32, 8, 64, 2, 2, 2) == 0
    small = lib.e2_workspace_bytes_ex(8, 32, 8, 64, 2, 2, 0)
    big = lib.e2_workspace_bytes_ex(8, 32, 8, 64, 2, 2, e2ga.E2_WS_LAYERED)
    assert big > small > 0
