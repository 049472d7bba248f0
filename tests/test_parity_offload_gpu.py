"""Parity of GPU-CPU offload in the cost model (Sec. 1; the plans' G--C
column, Sec. 4.3) with the oracle, through the C ABI.

Fleets drawn with a host side (half the devices unified, the others with
host RAM for offloaded blocks and a slower host rate and bandwidth): every
stage time, partition, T, Lambda and fitness bit-exact, and the G--C split of
every placed device equal to the oracle's device-memory block count for its
stage.
"""
import dataclasses

import numpy as np
import pytest

from oracle import oracle as O
from paper_2606_03770_gb300 import workloads as W

from test_parity_gpu import assert_eval_equal, assert_genomes_equal, engine, take

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()


def expected_gpu_layers(op, g, ora, K):
    """The oracle's device-memory blocks of every placed device."""
    P, M = g["perm"].shape
    out = np.full((P, M), -1, np.int16)
    for p in range(P):
        off = 0
        for c in range(int(g["nclus"][p])):
            m = int(g["sizes"][p, c])
            b = int(ora["bsel"][p, c])
            mu = int(ora["master"][p, c])
            for k in range(m):
                n = int(ora["layers"][p, off + k])
                if n >= 0 and b >= 0:
                    out[p, off + k] = op.gpu_blocks(b, int(g["perm"][p, off + k]), n, k == mu)
            off += m
    return out


CASES = [("c1_tiny", 64, 0, 0), ("c2", 1024, 0, 0), ("c2", 1024, 1, 0), ("c2", 512, 2, 1), ("c3", 256, 0, 0)]


@pytest.mark.parametrize("name,P,role_search,objective", CASES)
def test_offload_parity_full_population(name, P, role_search, objective):
    prob = dataclasses.replace(W.make_config(name, P=P, offload=True), role_search=role_search, objective=objective)
    eng = engine(prob)
    g = W.random_genomes(prob.M, prob.K_max, P, seed=23)
    eng.eval(g)
    gpu = eng.results()
    op = O.OracleProblem(prob)
    ora = op.eval_population(g, prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    g_eval = eng.get_population()                       # with the roles the search or rule chose
    assert np.array_equal(gpu["gpu_layers"], expected_gpu_layers(op, g_eval, ora, prob.K_max))
    st = eng.stats()
    assert st["paper_candidates"] == ora["cand"]
    assert st["served"] == int((ora["bsel"] >= 0).sum())
    # offloading is used: some placed device keeps part of its blocks in host memory
    placed = gpu["layers"] >= 0
    assert (gpu["gpu_layers"][placed] < gpu["layers"][placed]).any()
    eng.close()


@pytest.mark.parametrize("name,P,sample", [("c5", 8192, 128), ("c4", 16384, 48)])
def test_offload_full_size_sampled(name, P, sample):
    prob = W.make_config(name, P=P, offload=True)
    eng = engine(prob)
    eng.init_population(88)
    g = eng.get_population()
    eng.eval()
    gpu = eng.results()
    idx = np.sort(np.random.default_rng(8).choice(P, sample, replace=False))
    op = O.OracleProblem(prob)
    sub = take(g, idx)
    ora = op.eval_population(sub, prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora, rows=idx)
    assert np.array_equal(gpu["gpu_layers"][idx], expected_gpu_layers(op, sub, ora, prob.K_max))
    eng.close()


def test_without_offload_every_block_is_in_device_memory():
    prob = W.make_config("c2", P=256)
    eng = engine(prob)
    eng.init_population(3)
    eng.eval()
    gpu = eng.results()
    assert np.array_equal(gpu["gpu_layers"], gpu["layers"])
    eng.close()


def test_offload_generations():
    prob = W.make_config("c2", P=256, offload=True)
    ga = O.ga_of(prob)
    op = O.OracleProblem(prob)
    eng = engine(prob)
    eng.init_population(5)
    pop = O.init_population(ga, 5)
    for gen in range(1, 4):
        ora = op.eval_population(pop, prob.K_max, nthreads=O.num_threads())
        if gen % 2:
            eng.run_generation(5, gen)
        else:
            eng.eval(parts=False)
            eng.ga_step(5, gen)
        assert np.array_equal(eng.results()["fitness"], ora["fitness"]), gen
        pop = O.ga_step(ga, 5, gen, pop, ora["fitness"], O.elites(ga, pop, ora["fitness"]))
        assert_genomes_equal(eng.get_population(), pop)
    eng.close()
