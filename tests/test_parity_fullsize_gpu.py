"""Parity at the full sizes of the largest workloads, in the launch
configuration the benchmark uses (recorded generations on the full
population), against the oracle.

* 512 devices, 126 blocks, K_max 64, P 16,384: two generations, each with a
  256-genome evaluation sample recomputed by the oracle, the elites and the
  whole next population from the oracle's generation step (fed the GPU's
  fitness, whose sample was just checked bit for bit).
* 128 devices with congestion redrawn every generation, P 4,096: three
  generations of redraw -> evaluation -> step, each checked (the congestion
  matrix, a 256-genome sample under the new links, elites, next population).
"""
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


def test_largest_workload_two_generations():
    prob = W.make_config("c4")
    assert prob.P == 16384 and prob.M == 512 and prob.K_max == 64
    ga = O.ga_of(prob)
    op = O.OracleProblem(prob)
    eng = engine(prob)
    seed = 4242
    eng.init_population(seed)
    pop = O.init_population(ga, seed)
    rng = np.random.default_rng(17)
    for gen in (1, 2):
        assert_genomes_equal(eng.get_population(), pop)
        eng.run_generation(seed, gen)                 # the benchmark's recorded launch sequence
        gpu = eng.results()
        idx = np.sort(rng.choice(prob.P, 256, replace=False))
        ora = op.eval_population(take(pop, idx), prob.K_max, nthreads=O.num_threads())
        assert_eval_equal(gpu, ora, rows=idx)
        fit = gpu["fitness"]
        eidx = O.elites(ga, pop, fit)
        gi, gf = eng.elites()
        assert np.array_equal(gi, eidx) and np.array_equal(gf, fit[eidx])
        pop = O.ga_step(ga, seed, gen, pop, fit, eidx)
        assert_genomes_equal(eng.get_population(), pop)
    st = eng.stats()
    assert st["genomes"] == prob.P and st["dp_launches"] == 2
    eng.close()


def test_congestion_redraw_chain_three_generations():
    prob = W.make_config("c3")
    assert prob.P == 4096 and prob.redraw
    ga = O.ga_of(prob)
    eng = engine(prob)
    seed = 99
    eng.init_population(seed)
    pop = O.init_population(ga, seed)
    rng = np.random.default_rng(29)
    for gen in (1, 2, 3):
        assert_genomes_equal(eng.get_population(), pop)
        eng.redraw_congestion(seed, gen)
        cong = O.redraw_congestion(prob.M, seed, gen, prob.cong_lo, prob.cong_hi)
        assert np.array_equal(eng.congestion(), cong)
        eng.run_generation(seed, gen)
        gpu = eng.results()
        idx = np.sort(rng.choice(prob.P, 256, replace=False))
        ora = O.OracleProblem(prob, cong=cong).eval_population(take(pop, idx), prob.K_max,
                                                               nthreads=O.num_threads())
        assert_eval_equal(gpu, ora, rows=idx)
        fit = gpu["fitness"]
        eidx = O.elites(ga, pop, fit)
        assert np.array_equal(eng.elites()[0], eidx)
        pop = O.ga_step(ga, seed, gen, pop, fit, eidx)
        assert_genomes_equal(eng.get_population(), pop)
    eng.close()


def test_resume_from_a_saved_population_is_bit_exact():
    """Checkpoint and resume: ten generations straight equal five, the
    population saved to the host and loaded into a fresh context, five more
    (the generation's streams depend only on (seed, generation, slot), and
    the elites ride in slots [0, Q) of the population itself)."""
    prob = W.make_config("c2")
    seed = 7
    a = engine(prob)
    a.init_population(seed)
    for gen in range(1, 11):
        a.run_generation(seed, gen)
    straight = a.get_population()
    fit_straight = a.results()["fitness"]
    a.close()
    b = engine(prob)
    b.init_population(seed)
    for gen in range(1, 6):
        b.run_generation(seed, gen)
    saved = b.get_population()
    b.close()
    c = engine(prob)
    c.set_population(saved)
    for gen in range(6, 11):
        c.run_generation(seed, gen)
    assert_genomes_equal(c.get_population(), straight)
    assert np.array_equal(c.results()["fitness"], fit_straight)
    c.close()
