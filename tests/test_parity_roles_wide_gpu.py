"""Alg. 2's role search on genomes of up to 64 replicas, through the C ABI.

Only the replicas whose role is not fixed in the winning assignment are
enumerated (the others: a replica that serves neither role, and under the
waiting time one that cannot decode, whose roles the oracle's pins fix); a
genome with more than 20 such replicas keeps its own role bits and is
counted.  Against the oracle, whose search is pinned against the plain 2^R
enumeration.
"""
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


@pytest.mark.parametrize("name,P,sample,objective", [("c5", 8192, 128, 0), ("c5", 8192, 64, 1),
                                                      ("c4", 16384, 48, 0)])
def test_role_search_full_size_sampled(name, P, sample, objective):
    """The role search at the 32- and 64-replica workloads: the full population
    on the GPU, a sample by the oracle (all of it, including the capped count)."""
    prob = dataclasses.replace(W.make_config(name, P=P), role_search=1, objective=objective)
    eng = engine(prob)
    eng.init_population(61)
    g = eng.get_population()
    eng.eval()
    gpu = eng.results()
    idx = np.sort(np.random.default_rng(9).choice(P, sample, replace=False))
    ora = O.OracleProblem(prob).eval_population(take(g, idx), prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora, rows=idx)
    assert np.array_equal(eng.get_population()["roles"][idx], ora["roles"])
    st = eng.stats()
    # under the waiting time only replicas that can decode are enumerated, and
    # almost no genome has more than 20 of them; under the finishing time every
    # replica that serves either role is (a slow prefill replica can raise the
    # mean latency), so many more genomes are capped there
    if objective == 0:
        assert st["role_search_capped"] <= P // 100, st
    eng.close()


@pytest.mark.parametrize("objective", [0, 1])
def test_role_search_many_replicas_few_free(objective):
    """40 to 64 single- and multi-device replicas of which at most 20 can serve
    the free roles: the search runs over those; genomes with 21 to 26 are
    capped (own role bits).  Small-integer costs, so ties are frequent."""
    rng = np.random.default_rng(67 + objective)
    M, N, K, P = 96, 8, 64, 24
    prob = _edge_problem(rng, M, N, P, K, integer=True, Q=2, role_search=1, objective=objective, min_tps=0.02)
    # devices 0..31 have ample memory, the others too little to hold N blocks
    # alone, so a single-device replica of them serves nothing
    prob.mem = np.where(np.arange(M) < 32, 10 ** 6, 2).astype(np.uint64)
    g = dict(perm=np.zeros((P, M), np.uint16), sizes=np.zeros((P, K), np.uint16),
             nclus=np.zeros(P, np.uint8), roles=np.zeros(P, np.uint64))
    for p in range(P):                            # R - 1 single-device replicas, the last takes the rest
        R = int(rng.integers(40, 65))
        g["sizes"][p, :R] = 1
        g["sizes"][p, R - 1] = M - R + 1
        g["nclus"][p] = R
        g["roles"][p] = np.uint64(int(rng.integers(0, 1 << 62)) >> (62 - min(R, 62)))
    for p in range(P):                            # `want` strong devices alone in single-device replicas
        R = int(g["nclus"][p])
        want = int(rng.integers(8, 20)) if p % 3 else int(rng.integers(21, 27))
        strong = rng.permutation(32)
        weak = 32 + rng.permutation(M - 32)
        pos = np.sort(rng.choice(R - 1, want, replace=False))
        perm = np.empty(M, np.uint16)
        s_i = w_i = 0
        for c in range(R - 1):
            if s_i < want and c == pos[s_i]:
                perm[c] = strong[s_i]; s_i += 1
            else:
                perm[c] = weak[w_i]; w_i += 1
        rest = list(strong[s_i:]) + list(weak[w_i:])
        perm[R - 1:] = rest
        g["perm"][p] = perm
    eng = engine(prob)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, K, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    assert np.array_equal(eng.get_population()["roles"], ora["roles"])
    st = eng.stats()
    assert st["role_search_capped"] == ora["capped"]
    assert 0 < ora["capped"] < P
    eng.close()


def test_role_search_wide_generations():
    """Generations with the role search at K_max 32 (the 256-device fleet, a
    smaller population), recorded and separate calls alike."""
    prob = dataclasses.replace(W.make_config("c5", P=512), role_search=1)
    ga = O.ga_of(prob)
    op = O.OracleProblem(prob)
    eng = engine(prob)
    eng.init_population(13)
    pop = O.init_population(ga, 13)
    for gen in range(1, 4):
        ora = op.eval_population(pop, prob.K_max, nthreads=O.num_threads())
        if gen % 2:
            eng.run_generation(13, gen)
        else:
            eng.eval(parts=False)
            eng.ga_step(13, gen)
        assert np.array_equal(eng.results()["fitness"], ora["fitness"]), gen
        pop = dict(pop, roles=ora["roles"])
        pop = O.ga_step(ga, 13, gen, pop, ora["fitness"], O.elites(ga, pop, ora["fitness"]))
        assert_genomes_equal(eng.get_population(), pop)
    eng.close()
