"""Parity of the warp-per-run DP launch (the small replica sizes of a large
population, one DP run per warp) with the oracle, through the C ABI.

The second DP launch runs one run per warp when the population is large
enough (its slots at least eight times that launch's runs in flight) and no
four-warp launch of the small sizes raises the occupancy: the 80-block
workloads at full size.  Full populations (and role search, where each
replica runs in both roles) bit for bit, and a large population of
small-integer costs (many exact ties, memory walls, a Min_TPS floor) on which
every DP tie rule is exercised by the warp kernel.
"""
import dataclasses

import numpy as np
import pytest

from oracle import oracle as O
from paper_2606_03770_gb300 import workloads as W

from test_parity_gpu import _edge_problem, assert_eval_equal, assert_genomes_equal, engine

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()


def _warp_launch(st):
    assert st["dp_launches"] == 2 and st["dp_runs_per_cta_small"] == 4, st
    assert st["dp_runs_small"] > 0 and st["device_errors"] == 0, st


@pytest.mark.parametrize("name,P,role_search", [("c3", 4096, 0), ("c3", 2048, 1), ("c5", 1024, 0)])
def test_warp_launch_full_population(name, P, role_search):
    prob = dataclasses.replace(W.make_config(name, P=P), role_search=role_search)
    eng = engine(prob)
    g = W.random_genomes(prob.M, prob.K_max, P, seed=41)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    if role_search:
        assert np.array_equal(eng.get_population()["roles"], ora["roles"])
    st = eng.stats()
    _warp_launch(st)
    assert st["paper_candidates"] == ora["cand"]
    assert st["served"] == int((ora["bsel"] >= 0).sum())
    eng.close()


@pytest.mark.parametrize("min_tps", [0.0, 0.1])
def test_warp_launch_ties_and_memory_walls(min_tps):
    """Small-integer costs on 24 devices and 12 blocks (exact ties between
    splits, masters and batches; devices that cannot hold a block), 8,192
    genomes of up to six replicas: the whole population, then a generation."""
    rng = np.random.default_rng(77)
    M, N, K, P = 24, 12, 6, 8192
    prob = _edge_problem(rng, M, N, P, K, integer=True, Q=64, min_tps=min_tps)
    g = W.random_genomes(M, K, P, seed=13)
    eng = engine(prob)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, K, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    _warp_launch(eng.stats())
    assert np.isfinite(ora["T"]).sum() > 1000
    ga = O.ga_of(prob)
    eidx = O.elites(ga, g, gpu["fitness"])
    eng.ga_step(5, 1)
    assert_genomes_equal(eng.get_population(), O.ga_step(ga, 5, 1, g, gpu["fitness"], eidx))
    eng.close()


def test_small_population_keeps_one_launch():
    """At 1,024 genomes of the 32-device workload the runs per warp would be
    few: the small sizes stay in the four-warp launch."""
    prob = W.make_config("c2")
    eng = engine(prob)
    eng.init_population(3)
    eng.eval()
    st = eng.stats()
    assert st["dp_runs_per_cta_small"] in (0, 1), st
    eng.close()
