"""Parity of the comparison objectives of the paper's evaluation (Sec. 4.2,
"Baseline chosen") with the oracle, through the C ABI.

* objective 1: the per-request finishing time FT that HexGen-2 minimises, in
  place of the waiting time of Eq. 3-5 (with the genome's role bits, and with
  Alg. 2's brute-force role search);
* role_search 2: the adapted-SplitWise rule, the strongest replicas prefill
  (with either objective).

Bit-exact like the main parity suite: fitness, partitions, T, Lambda, the
roles written into the genomes, and whole next populations.
"""
import dataclasses

import numpy as np
import pytest

from oracle import oracle as O
from paper_2606_03770_gb300 import workloads as W

from test_parity_gpu import _edge_problem, _genomes_from, assert_eval_equal, assert_genomes_equal, engine, take

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()


CASES = [("c1_tiny", 64, 0, 1), ("c2", 1024, 0, 1), ("c1_tiny", 64, 1, 1), ("c2", 1024, 1, 1), ("c3", 256, 1, 1),
         ("c1_tiny", 64, 2, 0), ("c2", 1024, 2, 0), ("c2", 1024, 2, 1), ("c3", 512, 2, 1)]


@pytest.mark.parametrize("name,P,role_search,objective", CASES)
def test_objective_parity_full_population(name, P, role_search, objective):
    prob = dataclasses.replace(W.make_config(name, P=P), role_search=role_search, objective=objective)
    eng = engine(prob)
    g = W.random_genomes(prob.M, prob.K_max, P, seed=17 + role_search)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    assert np.array_equal(eng.get_population()["roles"], ora["roles"])
    st = eng.stats()
    assert st["paper_candidates"] == ora["cand"]
    assert st["served"] == int((ora["bsel"] >= 0).sum())
    assert np.isfinite(ora["fitness"][:, 0]).sum() >= min(P // 8, 20)
    eng.close()


@pytest.mark.parametrize("name,P,sample", [("c5", 8192, 128), ("c4", 16384, 48)])
def test_splitwise_full_size_sampled(name, P, sample):
    """The adapted-SplitWise rule at the sizes it is meant for (up to 32 and 64
    replicas per genome), full population on the GPU, a sample by the oracle."""
    prob = dataclasses.replace(W.make_config(name, P=P), role_search=2)
    eng = engine(prob)
    eng.init_population(77)
    g = eng.get_population()
    eng.eval()
    gpu = eng.results()
    idx = np.sort(np.random.default_rng(6).choice(P, sample, replace=False))
    ora = O.OracleProblem(prob).eval_population(take(g, idx), prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora, rows=idx)
    assert np.array_equal(eng.get_population()["roles"][idx], ora["roles"])
    eng.close()


@pytest.mark.parametrize("integer", [True, False])
def test_finishing_time_role_search_twenty_replicas(integer):
    """Alg. 2's role search under the finishing time: 9 to 20 replicas (up to
    2^20 assignments, each scored exactly), against the oracle's plain
    enumeration."""
    rng = np.random.default_rng(53 + integer)
    M, N, K, P = 40, 24, 20, 16
    prob = _edge_problem(rng, M, N, P, K, integer=integer, Q=2, role_search=1, objective=1,
                         min_tps=0.05 if integer else 1e-5)
    groups = []
    for p in range(P):
        R = int(rng.integers(9, 21))
        cuts = np.sort(rng.choice(np.arange(1, M), R - 1, replace=False))
        groups.append(list(np.diff(np.concatenate([[0], cuts, [M]])).astype(int)))
    g = _genomes_from(M, K, groups, rng)
    eng = engine(prob)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, K, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    assert np.array_equal(eng.get_population()["roles"], ora["roles"])
    assert np.isfinite(ora["fitness"][:, 0]).all()
    eng.close()


@pytest.mark.parametrize("role_search,objective", [(2, 1), (2, 0), (1, 1), (0, 1)])
def test_objective_generations(role_search, objective):
    """Generations under the comparison objectives, recorded and separate
    calls alike, against the oracle (whose population takes the roles the
    rule or the search chose)."""
    prob = dataclasses.replace(W.make_config("c2", P=256), role_search=role_search, objective=objective)
    ga = O.ga_of(prob)
    op = O.OracleProblem(prob)
    eng = engine(prob)
    eng.init_population(21)
    pop = O.init_population(ga, 21)
    for gen in range(1, 5):
        ora = op.eval_population(pop, prob.K_max, nthreads=O.num_threads())
        if gen % 2:
            eng.run_generation(21, gen)
        else:
            eng.eval(parts=False)
            eng.ga_step(21, gen)
        assert np.array_equal(eng.results()["fitness"], ora["fitness"]), gen
        pop = dict(pop, roles=ora["roles"])
        pop = O.ga_step(ga, 21, gen, pop, ora["fitness"], O.elites(ga, pop, ora["fitness"]))
        assert_genomes_equal(eng.get_population(), pop)
    eng.close()
