"""Parity of the CUDA path with the CPU oracle, through the C ABI.

Bit-exact: genomes, partitions (blocks per device, master, decode batch),
stage bottleneck T, latency Lambda and fitness (w, phase, PS, DS): the kernels
and the oracle perform the same IEEE-754 float64 operations in the same order
with no fused multiply-add, so the benchmark spec's tolerance (1e-12 relative on
fitness) is met with equality, which the genetic algorithm needs anyway
(selection compares fitness).
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2606_03770_gb300 import workloads as W

pytestmark = pytest.mark.gpu

FIELDS = ("layers", "master", "bsel", "T", "L")


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as ge
    ge.build()


def engine(prob):
    from paper_2606_03770_gb300.e2ga import Engine
    return Engine(prob)


def assert_eval_equal(gpu, ora, rows=None):
    rows = slice(None) if rows is None else rows
    for k in FIELDS:
        a, b = gpu[k][rows], ora[k]
        assert np.array_equal(a, b), (k, np.argwhere(a != b)[:5])
    fa, fb = gpu["fitness"][rows], ora["fitness"]
    assert np.array_equal(fa, fb), np.argwhere(fa != fb)[:5]
    # the stated tolerance, for the record
    fin = np.isfinite(fb)
    assert np.all(np.abs(fa[fin] - fb[fin]) <= 1e-12 * np.abs(fb[fin]))


def take(g, idx):
    return {k: np.ascontiguousarray(v[idx]) for k, v in g.items()}


@pytest.mark.parametrize("name,P", [("c1_tiny", 64), ("c2", 1024)])
def test_eval_parity_full_population(name, P):
    prob = W.make_config(name, P=P)
    eng = engine(prob)
    g = W.random_genomes(prob.M, prob.K_max, P, seed=11)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    st = eng.stats()
    assert st["genomes"] == P and st["replicas"] == int(g["nclus"].sum())
    assert st["paper_candidates"] == ora["cand"]
    assert st["served"] == int((ora["bsel"] >= 0).sum())
    eng.close()


@pytest.mark.parametrize("name,P,sample", [("c3", 4096, 256), ("c5", 8192, 256), ("c4", 16384, 32)])
def test_eval_parity_full_size_sampled(name, P, sample):
    """Full-size population on the GPU (the benchmark's launch shape); a seeded
    sample of genomes recomputed one by one by the oracle."""
    prob = W.make_config(name, P=P)
    eng = engine(prob)
    eng.init_population(2024)
    eng.eval()
    gpu = eng.results()
    g = eng.get_population()
    idx = np.sort(np.random.default_rng(5).choice(P, sample, replace=False))
    ora = O.OracleProblem(prob).eval_population(take(g, idx), prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora, rows=idx)
    # the 126-block model's largest DP spills its suffix columns to a global
    # scratch (6 CTAs per SM instead of 4); the small replica sizes run in a
    # second launch that does not spill, at that kernel's best occupancy
    st = eng.stats()
    assert st["dp_launches"] == (2 if st["dp_ctas_small"] else 1)
    assert (st["dp_runs_small"] > 0) == (st["dp_launches"] == 2), st
    if name == "c4":
        assert st["dp_launches"] == 2 and st["dp_ctas_small"] > st["dp_ctas"], st
        assert st["dp_smem_small"] < st["dp_smem"] <= 40 * 1024, st
    eng.close()


def test_init_population_parity():
    for name, P in (("c1_tiny", 64), ("c2", 1024), ("c4", 2048)):
        prob = W.make_config(name, P=P)
        eng = engine(prob)
        eng.init_population(99)
        got = eng.get_population()
        ref = O.init_population(O.ga_of(prob), 99)
        for k in ref:
            assert np.array_equal(got[k], ref[k]), (name, k)
        eng.close()


@pytest.mark.parametrize("name,P,gens,check_eval", [("c1_tiny", 64, 6, True), ("c2", 1024, 4, True),
                                                    ("c5", 8192, 2, False)])
def test_ga_generations_parity(name, P, gens, check_eval):
    """Every generation: GPU fitness (checked against the oracle where cheap,
    sampled otherwise), elites, and the whole next population bit-exact."""
    prob = W.make_config(name, P=P)
    ga = O.ga_of(prob)
    op = O.OracleProblem(prob)
    eng = engine(prob)
    seed = 314
    eng.init_population(seed)
    pop = O.init_population(ga, seed)
    for gen in range(1, gens + 1):
        assert_genomes_equal(eng.get_population(), pop)
        eng.eval()
        gpu = eng.results()
        if check_eval:
            ora = op.eval_population(pop, prob.K_max, nthreads=O.num_threads())
            assert_eval_equal(gpu, ora)
        else:
            idx = np.sort(np.random.default_rng(gen).choice(P, 64, replace=False))
            ora = op.eval_population(take(pop, idx), prob.K_max, nthreads=O.num_threads())
            assert_eval_equal(gpu, ora, rows=idx)
        fit = gpu["fitness"]
        eidx = O.elites(ga, pop, fit)
        eng.ga_step(seed, gen)
        gi, gf = eng.elites()
        assert np.array_equal(gi, eidx)
        assert np.array_equal(gf, fit[eidx])
        pop = O.ga_step(ga, seed, gen, pop, fit, eidx)
    assert_genomes_equal(eng.get_population(), pop)
    eng.close()


def assert_genomes_equal(a, b):
    for k in ("perm", "sizes", "nclus", "roles"):
        assert np.array_equal(a[k], b[k]), (k, np.argwhere(a[k] != b[k])[:5])


def test_congestion_redraw_parity():
    prob = W.make_config("c3", P=512)
    eng = engine(prob)
    for gen in (1, 2, 7):
        eng.redraw_congestion(77, gen)
        c = eng.congestion()
        ref = O.redraw_congestion(prob.M, 77, gen, prob.cong_lo, prob.cong_hi)
        assert np.array_equal(c, ref)
    eng.init_population(5)
    eng.eval()
    gpu = eng.results()
    g = eng.get_population()
    idx = np.arange(0, 512, 4)
    ora = O.OracleProblem(prob, cong=ref).eval_population(take(g, idx), prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora, rows=idx)
    eng.close()


def _edge_problem(rng, M, N, P, K, integer=True, **kw):
    from test_oracle_pins import tiny_problem
    p = tiny_problem(rng, M, N, V=4, integer=integer)
    p.P, p.K_max, p.Q = P, K, kw.pop("Q", 1)
    for k, v in kw.items():
        setattr(p, k, v)
    return p


@pytest.mark.parametrize("case", range(12))
def test_eval_parity_edge_cases(case):
    """Ties (small-integer costs), memory walls, replicas larger than the model
    (m > N), single-device replicas, one replica, a ragged population."""
    rng = np.random.default_rng(1000 + case)
    M = [3, 6, 9, 12, 7, 5, 16, 40, 8, 2, 33, 1][case]
    N = [2, 5, 4, 12, 30, 1, 9, 20, 8, 7, 64, 3][case]
    K = min(M, [1, 3, 8, 4, 7, 2, 16, 12, 8, 2, 33, 1][case])
    P = [1, 37, 100, 129, 255, 17, 300, 64, 513, 9, 70, 5][case]
    prob = _edge_problem(rng, M, N, P, K, integer=case % 3 != 2, Q=min(P, 3), min_tps=0.05 * (case % 4))
    g = W.random_genomes(M, K, P, seed=case)
    eng = engine(prob)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, K, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    assert eng.stats()["paper_candidates"] == ora["cand"]
    # a generation step on these odd shapes too
    ga = O.ga_of(prob)
    eidx = O.elites(ga, g, gpu["fitness"])
    eng.ga_step(3, 1)
    assert_genomes_equal(eng.get_population(), O.ga_step(ga, 3, 1, g, gpu["fitness"], eidx))
    eng.close()


@pytest.mark.parametrize("min_tps", [0.0, 0.02])
def test_spilled_layout_tie_heavy(min_tps):
    """Replicas of ~20 devices over a 126-block model run in the spilled layout,
    where the prefix chain speculates on the head on device 1: small-integer
    costs make the master-free optimum, V_1 and the other masters tie often, so
    both the proof of mu* = 1 and its fallback (the chain again without the
    head, the combine seeded with master 1) meet exact ties."""
    rng = np.random.default_rng(606)
    M, N, K, P = 64, 126, 3, 64
    prob = _edge_problem(rng, M, N, P, K, integer=True, Q=4, min_tps=min_tps)
    g = W.random_genomes(M, K, P, seed=66)
    eng = engine(prob)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, K, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    st = eng.stats()
    assert st["dp_smem"] <= 40 * 1024 and st["device_errors"] == 0, st   # the spilled layout
    assert st["served"] == int((ora["bsel"] >= 0).sum()) > 20
    eng.close()


@pytest.mark.parametrize("case", range(6))
def test_eval_parity_costs_growing_with_batch(case):
    """The small-integer edge problems with each decode cost row sorted, so
    that costs grow with the batch (ties between batches included): the
    pre-pass then searches its monotone memory and latency tests instead of
    testing every batch, with exact ties and memory walls at every step."""
    rng = np.random.default_rng(2000 + case)
    M, N, K, P = [(6, 5, 3, 40), (12, 12, 4, 129), (7, 30, 7, 255), (16, 9, 16, 300), (8, 8, 8, 513),
                  (33, 64, 33, 70)][case]
    prob = _edge_problem(rng, M, N, P, K, integer=case % 3 != 2, Q=3, min_tps=0.05 * (case % 4 + 1))
    for f in ("blk_flops", "blk_bytes", "blk_mem", "head_flops", "head_bytes", "head_mem", "act_bytes"):
        row = np.asarray(getattr(prob, f)).copy()       # prefill, then 8 decode batches drawn from the rows
        row = np.concatenate([row[:1], rng.choice(row[1:], 8)])
        row[1:] = np.sort(row[1:])
        setattr(prob, f, row)
    assert prob.b_max == 8
    g = W.random_genomes(M, K, P, seed=case)
    eng = engine(prob)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, K, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    st = eng.stats()
    assert st["paper_candidates"] == ora["cand"]
    assert st["served"] == int((ora["bsel"] >= 0).sum())
    eng.close()


def test_elites_with_duplicates_and_Q_extremes():
    prob = W.make_config("c1_tiny", P=96)
    g = W.random_genomes(prob.M, prob.K_max, 96, seed=4)
    for dst, src in [(10, 3), (11, 3), (40, 12), (95, 0)]:
        for k in g:
            g[k][dst] = g[k][src]
    for Q in (0, 1, 5, 96):
        prob.Q = Q
        eng = engine(prob)
        eng.eval(g)
        fit = eng.results()["fitness"]
        ga = O.ga_of(prob)
        eidx = O.elites(ga, g, fit)
        eng.ga_step(8, 2)
        if Q:
            gi, _ = eng.elites()
            assert np.array_equal(gi, eidx)
        assert_genomes_equal(eng.get_population(), O.ga_step(ga, 8, 2, g, fit, eidx))
        eng.close()


@pytest.mark.parametrize("P,Q", [(5000, 157), (8200, 8200)])
def test_elites_large_population_with_duplicates(P, Q):
    """Populations of several thousand genomes (many tiles of the duplicate
    test and the ranks): a ragged size, many planted duplicates (copies of a
    few genomes spread over the population, ties in every key), Q = ceil(P/32)
    and Q = P; elites and next population against the oracle."""
    prob = W.make_config("c1_tiny", P=P)
    prob.Q = Q
    rng = np.random.default_rng(17)
    g = W.random_genomes(prob.M, prob.K_max, P, seed=5)
    src = rng.integers(0, 50, 600)
    dst = rng.choice(np.arange(50, P), 600, replace=False)
    for a, b in zip(dst, src):
        for k in g:
            g[k][a] = g[k][b]
    eng = engine(prob)
    eng.eval(g)
    fit = eng.results()["fitness"]
    ga = O.ga_of(prob)
    eidx = O.elites(ga, g, fit)
    eng.ga_step(8, 3)
    gi, gf = eng.elites()
    assert np.array_equal(gi, eidx)
    assert np.array_equal(gf, fit[eidx])
    assert_genomes_equal(eng.get_population(), O.ga_step(ga, 8, 3, g, fit, eidx))
    eng.close()


def test_host_and_device_buffers_agree():
    import torch
    prob = W.make_config("c1_tiny", P=64)
    g = W.random_genomes(prob.M, prob.K_max, 64, seed=2)
    eng = engine(prob)
    host_fit = np.zeros((64, 4))
    eng.eval(g, fitness=host_fit)                     # host genomes, host output
    dg = {k: torch.from_numpy(v.astype(np.int16 if v.dtype == np.uint16 else v.dtype)).cuda()
          if v.dtype != np.uint64 else torch.from_numpy(v.view(np.int64)).cuda() for k, v in g.items()}
    dev_fit = torch.empty((64, 4), dtype=torch.float64, device="cuda")
    eng.eval(dg, fitness=dev_fit)                     # device genomes, device output
    assert np.array_equal(host_fit, dev_fit.cpu().numpy())
    eng.close()


def test_errors_are_statuses_not_faults():
    from paper_2606_03770_gb300 import e2ga
    prob = W.make_config("c1_tiny", P=8)
    eng = engine(prob)
    with pytest.raises(e2ga.E2Error) as ei:
        eng.ga_step(1, 1)                             # nothing evaluated yet
    assert ei.value.status == e2ga.E2_ESTATE
    g = W.random_genomes(prob.M, prob.K_max, 8, seed=1)
    bad = {k: v.copy() for k, v in g.items()}
    bad["perm"][5, 0] = bad["perm"][5, 1]             # not a permutation
    with pytest.raises(e2ga.E2Error) as ei:
        eng.set_population(bad)
    assert ei.value.status == e2ga.E2_EINVAL and "genome 5" in str(ei.value)
    bad = {k: v.copy() for k, v in g.items()}
    bad["sizes"][2, :] = 0                            # sizes do not sum to M
    with pytest.raises(e2ga.E2Error):
        eng.eval(bad)
    eng.eval(g)                                       # the context is still usable
    assert np.isfinite(eng.results()["T"]).any()
    eng.close()


def test_dp_timing_events_bracket_the_dp_kernel():
    import torch
    from paper_2606_03770_gb300 import e2ga
    prob = W.make_config("c2", P=256)
    g = W.random_genomes(prob.M, prob.K_max, 256, seed=4)
    eng = engine(prob)
    stream = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    x, y = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for e in (x, y):
        e.record(stream)                              # creates the CUDA events
    with pytest.raises(e2ga.E2Error):
        eng.set_timing_events(x, None)                # one event alone is rejected
    eng.set_timing_events(x, y)
    eng.set_population(g)
    a.record(stream)
    eng.eval(parts=False)
    b.record(stream)
    torch.cuda.synchronize()
    dp, whole = x.elapsed_time(y), a.elapsed_time(b)
    assert 0 < dp <= whole
    eng.set_timing_events()                           # hook off: the events are not touched again
    eng.eval(g)
    torch.cuda.synchronize()
    assert x.elapsed_time(y) == dp
    eng.close()


def test_min_tps_boundary_exact():
    """Min_TPS set to exactly 1.0 / Lambda of a serving decode replica, then to
    the next double above it: the decode test of Alg. 2 flips for that replica
    exactly as the oracle's division-based test does."""
    import dataclasses
    import math
    prob = W.make_config("c2", P=256)
    g = W.random_genomes(prob.M, prob.K_max, 256, seed=21)
    ora = O.OracleProblem(prob).eval_population(g, prob.K_max, nthreads=O.num_threads())
    cand = [(p, c) for p in range(256) for c in range(int(g["nclus"][p]))
            if (int(g["roles"][p]) >> c) & 1 and ora["bsel"][p, c] >= 1]
    assert cand
    p, c = cand[len(cand) // 2]
    lam = float(ora["L"][p, c])
    served = []
    for tps in (1.0 / lam, math.nextafter(1.0 / lam, math.inf)):
        pb = dataclasses.replace(prob, min_tps=tps)
        eng = engine(pb)
        eng.eval(g)
        gpu = eng.results()
        ref = O.OracleProblem(pb).eval_population(g, prob.K_max, nthreads=O.num_threads())
        assert_eval_equal(gpu, ref)
        served.append(int(ref["bsel"][p, c]))
        eng.close()
    assert served[0] == ora["bsel"][p, c] and served[1] != served[0]


@pytest.mark.parametrize("name,P,gens", [("c1_tiny", 64, 5), ("c2", 1024, 5), ("c4", 1024, 4), ("c5", 4096, 3)])
def test_recorded_generation_matches_separate_calls(name, P, gens):
    """e2_run_generation (one recorded graph per population buffer) gives the
    populations and fitness of e2_eval_population + e2_ga_step, also when
    interleaved with the separate calls and after the timing events change."""
    import torch
    prob = W.make_config(name, P=P)
    a, b = engine(prob), engine(prob)
    a.init_population(5)
    b.init_population(5)
    x, y = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for e in (x, y):
        e.record(torch.cuda.current_stream())
    for gen in range(1, gens + 1):
        la, lb = a.stats()["launches"], b.stats()["launches"]
        a.eval(parts=False)
        fa = a.results()["fitness"]
        a.ga_step(5, gen)
        if gen == 3:                                   # the separate calls on the recording engine
            b.eval(parts=False)
            fb = b.results()["fitness"]
            b.ga_step(5, gen)
        else:
            if gen == 4:
                b.set_timing_events(x, y)              # recorded again, with the events
            b.run_generation(5, gen)
            fb = b.results()["fitness"]
        assert np.array_equal(fa, fb), gen
        assert_genomes_equal(a.get_population(), b.get_population())
        # a replay counts the recorded kernel nodes: as many as the separate calls launch
        # (pre-pass, bin scan, scatter, DP launches, finaliser, duplicates -- from 4,096
        # genomes a fingerprint table and a lookup --, elite selection, candidate ranks,
        # full ranks, children)
        sa, sb = a.stats(), b.stats()
        expected = 9 + sa["dp_launches"] + (1 if P >= 4096 else 0)
        assert sa["launches"] - la == sb["launches"] - lb == expected, gen
    torch.cuda.synchronize()
    assert x.elapsed_time(y) > 0
    b.set_timing_events()
    a.close()
    b.close()


def test_generation_io_matches_separate_calls():
    """e2_run_generation_io (population in, one generation, fitness and next
    population out, one synchronisation) gives what e2_set_population +
    e2_run_generation + e2_get_results + e2_get_population give, with host
    arrays and with device arrays, and chains over generations."""
    import torch
    prob = W.make_config("c2", P=512)
    a, b = engine(prob), engine(prob)
    g = W.random_genomes(prob.M, prob.K_max, prob.P, seed=21)
    cur = {k: v.copy() for k, v in g.items()}
    for gen in range(1, 5):
        a.set_population(cur)
        a.run_generation(9, gen)
        fa = a.results()["fitness"]
        na = a.get_population()
        if gen % 2:                                    # host arrays
            fb = np.zeros((prob.P, 4), np.float64)
            nb = {k: np.zeros_like(v) for k, v in cur.items()}
            b.run_generation_io(9, gen, population=cur, fitness=fb, next_out=nb)
        else:                                          # device arrays
            dev = {k: torch.from_numpy(v.view(np.int16) if v.dtype == np.uint16 else
                                       v.view(np.int64) if v.dtype == np.uint64 else v).cuda()
                   for k, v in cur.items()}
            fd = torch.zeros((prob.P, 4), dtype=torch.float64, device="cuda")
            nd = {k: torch.empty_like(t) for k, t in dev.items()}
            b.run_generation_io(9, gen, population=dev, fitness=fd, next_out=nd)
            torch.cuda.synchronize()
            fb = fd.cpu().numpy()
            nb = {k: nd[k].cpu().numpy().view(cur[k].dtype) for k in cur}
        assert np.array_equal(fa, fb), gen
        assert_genomes_equal(na, nb)
        cur = nb
    # chained without an upload: the context's own next population
    a.run_generation(9, 5)
    fb = np.zeros((prob.P, 4), np.float64)
    b.run_generation_io(9, 5, fitness=fb)
    assert np.array_equal(a.results()["fitness"], fb)
    a.close()
    b.close()


def test_generation_io_invalid_genome_is_replaced():
    """An invalid genome in the uploaded population: E2_EINVAL naming it, the
    generation ran with it replaced by the identity ordering as one prefill
    replica, and the context stays usable."""
    from paper_2606_03770_gb300 import e2ga
    prob = W.make_config("c1_tiny", P=16)
    eng = engine(prob)
    g = W.random_genomes(prob.M, prob.K_max, prob.P, seed=4)
    bad = {k: v.copy() for k, v in g.items()}
    bad["perm"][7, 2] = bad["perm"][7, 3]
    fit = np.zeros((prob.P, 4), np.float64)
    with pytest.raises(e2ga.E2Error) as ei:
        eng.run_generation_io(3, 1, population=bad, fitness=fit)
    assert ei.value.status == e2ga.E2_EINVAL and "genome 7" in str(ei.value)
    fixed = {k: v.copy() for k, v in g.items()}
    fixed["perm"][7] = np.arange(prob.M)
    fixed["sizes"][7] = 0
    fixed["sizes"][7, 0] = prob.M
    fixed["nclus"][7] = 1
    fixed["roles"][7] = 0
    ora = O.OracleProblem(prob).eval_population(fixed, prob.K_max, nthreads=O.num_threads())
    assert np.array_equal(fit, ora["fitness"])
    # the same replacement by e2_set_population; then evaluation is safe
    with pytest.raises(e2ga.E2Error):
        eng.set_population(bad)
    assert_genomes_equal(eng.get_population(), fixed)
    eng.eval()
    assert np.array_equal(eng.results()["fitness"], ora["fitness"])
    eng.close()


@pytest.mark.parametrize("name,P", [("c1_tiny", 64), ("c2", 1024), ("c3", 256)])
def test_role_search_parity(name, P):
    """Alg. 2's brute-force role assignment: every replica evaluated in both
    roles, the best of the 2^R assignments chosen and written into the
    genomes; compared with the oracle element by element."""
    import dataclasses
    prob = dataclasses.replace(W.make_config(name, P=P), role_search=1)
    eng = engine(prob)
    g = W.random_genomes(prob.M, prob.K_max, P, seed=13)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, prob.K_max, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    assert np.array_equal(eng.get_population()["roles"], ora["roles"])
    st = eng.stats()
    assert st["paper_candidates"] == ora["cand"]
    assert st["served"] == int((ora["bsel"] >= 0).sum())
    eng.close()


@pytest.mark.parametrize("integer,kw", [(True, dict(min_tps=0.05)), (True, dict(min_tps=0.05, t_a=100.0)),
                                        (False, dict(min_tps=1e-5)), (False, dict(min_tps=1e-6, t_a=1e4))])
def test_role_search_twenty_replicas(integer, kw):
    """The largest role search the ABI takes: genomes of 9 to 20 replicas (up
    to 2^20 assignments, walked in Gray-code order with screens), small-integer
    or fractional costs, with w > 0 or on the w = 0 plateau (a large T_a),
    where the phase decides; against the oracle's plain enumeration."""
    rng = np.random.default_rng(31 + integer)
    M, N, K, P = 40, 24, 20, 24
    prob = _edge_problem(rng, M, N, P, K, integer=integer, Q=2, role_search=1, **kw)
    groups = []
    for p in range(P):
        R = int(rng.integers(9, 21)) if p % 3 == 0 else int(rng.integers(17, 21))
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
    assert (ora["fitness"][:, 0] == 0).any() == ("t_a" in kw)
    eng.close()


def test_role_search_with_two_dp_launches():
    """The role search on a fleet whose DP runs in two shared-memory classes
    (220-block rows): both roles of every replica through both launches."""
    rng = np.random.default_rng(41)
    M, N, K, P = 48, 220, 8, 24
    prob = _edge_problem(rng, M, N, P, K, integer=True, Q=2, min_tps=0.01, role_search=1)
    g = W.random_genomes(M, K, P, seed=9)
    eng = engine(prob)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, K, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    assert np.array_equal(eng.get_population()["roles"], ora["roles"])
    st = eng.stats()
    assert st["dp_launches"] == 2 and 0 < st["dp_runs_small"] < st["dp_runs"], st
    eng.close()


def test_role_search_generations():
    """Generations with the role search, recorded and separate calls alike,
    against the oracle (whose population takes the roles it chose)."""
    import dataclasses
    prob = dataclasses.replace(W.make_config("c2", P=256), role_search=1)
    ga = O.ga_of(prob)
    op = O.OracleProblem(prob)
    eng = engine(prob)
    eng.init_population(9)
    pop = O.init_population(ga, 9)
    assert_genomes_equal(eng.get_population(), pop)
    for gen in range(1, 5):
        ora = op.eval_population(pop, prob.K_max, nthreads=O.num_threads())
        if gen % 2:
            eng.run_generation(9, gen)
        else:
            eng.eval(parts=False)
            eng.ga_step(9, gen)
        assert np.array_equal(eng.results()["fitness"], ora["fitness"]), gen
        pop = dict(pop, roles=ora["roles"])
        pop = O.ga_step(ga, 9, gen, pop, ora["fitness"], O.elites(ga, pop, ora["fitness"]))
        assert_genomes_equal(eng.get_population(), pop)
    eng.close()


def _genomes_from(M, K, groups, rng):
    """Genomes with the given replica sizes (one list per genome) over random orderings."""
    P = len(groups)
    g = dict(perm=np.zeros((P, M), np.uint16), sizes=np.zeros((P, K), np.uint16),
             nclus=np.zeros(P, np.uint8), roles=np.zeros(P, np.uint64))
    for p, sz in enumerate(groups):
        assert sum(sz) == M and len(sz) <= K
        g["perm"][p] = rng.permutation(M)
        g["sizes"][p, :len(sz)] = sz
        g["nclus"][p] = len(sz)
        g["roles"][p] = rng.integers(0, 1 << len(sz))
    return g


@pytest.mark.parametrize("case", ["wide rows", "largest replica"])
def test_eval_parity_maximum_sizes(case):
    """The largest shapes the ABI takes: cost rows of ~300 blocks (W > 256,
    ~190 KB of DP shared memory), and a replica of 256 devices (the limit) next
    to mixed ones; then a generation step on them."""
    rng = np.random.default_rng(77)
    if case == "wide rows":
        M, N, K = 64, 300, 6
        prob = _edge_problem(rng, M, N, 12, K, integer=False, Q=2, min_tps=0.02)
        g = W.random_genomes(M, K, 12, seed=5)
    else:
        M, N, K = 256, 260, 2
        prob = _edge_problem(rng, M, N, 3, K, integer=True, Q=1, min_tps=0.01)
        g = _genomes_from(M, K, [[256], [250, 6], [200, 56]], rng)
    eng = engine(prob)
    eng.eval(g)
    gpu = eng.results()
    ora = O.OracleProblem(prob).eval_population(g, K, nthreads=O.num_threads())
    assert_eval_equal(gpu, ora)
    st = eng.stats()
    assert st["paper_candidates"] == ora["cand"]
    if case != "wide rows":
        # replicas of 6, 250 and 256 devices (W <= 255 with few devices, or a
        # short row) need less than half the shared memory of the 56- and
        # 200-device ones: they run in the second DP launch
        assert st["dp_launches"] == 2 and 0 < st["dp_runs_small"] <= st["dp_runs"], st
    assert np.isfinite(ora["T"]).any()
    ga = O.ga_of(prob)
    eidx = O.elites(ga, g, ora["fitness"])
    eng.ga_step(3, 1)
    assert_genomes_equal(eng.get_population(), O.ga_step(ga, 3, 1, g, ora["fitness"], eidx))
    eng.close()
