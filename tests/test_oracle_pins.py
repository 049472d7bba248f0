"""Pins for the CPU oracle: it is checked against what the paper and the
mathematics fix, never against itself.

* brute force over every composition of the blocks and every master (DP value,
  master, partition under the smallest-split tie rule);
* closed forms (identical devices, free links: ceil(N/m) blocks on the slowest
  stage; the canonical split 3,3,4 of 10 blocks on 3 devices);
* the paper's worked examples (20 kB over 100 Mbps = 1.6 ms; the gene
  [(0..5),(3,1,2)]);
* hand-computed stage costs and objective values (Eq. 3-5);
* invariants of the formulation (blocks sum to N, >= 1 per device, memory fits,
  the bottleneck recomputed from the partition equals the DP value);
* exact metamorphic scaling by powers of two;
* Philox-4x32-10 known-answer vectors; GA operator validity and frequencies.
"""
import itertools
import math
import os

import numpy as np
import pytest

from oracle import oracle as O
from paper_2606_03770_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
INF = math.inf


# ---------------------------------------------------------------------------
# helpers
# ---------------------------------------------------------------------------
def tiny_problem(rng, M, N, V=3, integer=True, tight_mem=True, head=True):
    """Small problem whose costs are small integers / simple ratios, so that
    the DP has many exact ties, memory walls and links that dominate."""
    if integer:
        rate = rng.choice([1.0, 2.0, 4.0, 0.5], M)
        bw = rng.choice([1.0, 2.0, 8.0], M)
        blk_flops = rng.integers(1, 4, V)
        blk_bytes = rng.integers(0, 4, V)
    else:
        rate = rng.uniform(0.5, 3.0, M)
        bw = rng.uniform(0.5, 3.0, M)
        blk_flops = rng.integers(1, 1000, V)
        blk_bytes = rng.integers(0, 1000, V)
    blk_mem = rng.integers(1, 3, V)
    mem = rng.integers(N // 2 if tight_mem else 4 * N, 4 * N + 3, M) if tight_mem else np.full(M, 10 * N)
    head_flops = rng.integers(0, 6, V) if head else np.zeros(V, int)
    head_bytes = rng.integers(0, 6, V) if head else np.zeros(V, int)
    head_mem = rng.integers(0, 3, V) if head else np.zeros(V, int)
    act = rng.integers(0, 4, V)
    link_bw = rng.choice([0.5, 1.0, 2.0, np.inf], (M, M))
    cong = rng.choice([0.5, 1.0], (M, M))
    return W.make_problem(rate, bw, mem, link_bw, cong, N, blk_flops, blk_bytes, blk_mem,
                          head_flops, head_bytes, head_mem, act, NP=64, ND=64)


def compositions(total, parts):
    """All (n_1..n_parts), n_t >= 1, sum = total."""
    for cuts in itertools.combinations(range(1, total), parts - 1):
        edges = (0,) + cuts + (total,)
        yield tuple(edges[t + 1] - edges[t] for t in range(parts))


def bf_value(op, v, devs, layers_total, k, mu):
    """min over compositions of layers_total blocks on devs[0..k) with master mu
    (0-based, may be >= k meaning 'not among them') of the largest stage or link."""
    best = INF
    for comp in compositions(layers_total, k):
        worst = 0.0
        for t in range(k):
            worst = max(worst, op.stage_cost(v, int(devs[t]), comp[t], t == mu))
            if t >= 1:
                worst = max(worst, op.link_cost(v, int(devs[t - 1]), int(devs[t])))
        best = min(best, worst)
    return best


def bf_dp(op, v, devs, N):
    """Brute-force DP_Pipe: value, first optimal master, and the partition the
    smallest-split tie rule selects (walk back from the last device; at each
    step the smallest start j that keeps the optimum, where the optimum of the
    prefix is again found by enumeration)."""
    m = len(devs)
    if m > N:
        return None
    vals = [bf_value(op, v, devs, N, m, mu) for mu in range(m)]
    V = min(vals)
    if V == INF:
        return None
    mu = vals.index(V)
    layers = [0] * m
    i = N - 1
    for k in range(m, 1, -1):
        target = bf_value(op, v, devs, i + 1, k, mu)
        tau = op.link_cost(v, int(devs[k - 2]), int(devs[k - 1]))
        for j in range(k - 1, i + 1):
            prev = bf_value(op, v, devs, j, k - 1, mu)
            c = max(prev, op.stage_cost(v, int(devs[k - 1]), i - j + 1, mu == k - 1), tau)
            if c == target:
                break
        layers[k - 1] = i - j + 1
        i = j - 1
    layers[0] = i + 1
    return V, mu, layers


# ---------------------------------------------------------------------------
# Philox
# ---------------------------------------------------------------------------
def test_philox_known_answers():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt"))
            if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = O.philox(v[0:4], v[4:6])
        assert [int(x) for x in out] == v[6:10]


def test_philox_stream_layout_and_uniformity():
    # word t of a stream is word t%4 of block t//4
    seed = 0x123456789ABCDEF
    blk = O.philox([5, 7, 3, 4], [seed & 0xFFFFFFFF, seed >> 32])
    assert [O.word(seed, 3, 7, 4, 20 + t) for t in range(4)] == [int(x) for x in blk]
    w = np.array([O.word(1, 0, 0, 0, t) for t in range(40000)], dtype=np.float64)
    u = w / 2.0 ** 32
    assert abs(u.mean() - 0.5) < 0.01 and abs(u.var() - 1 / 12) < 0.005


def test_threshold():
    assert O.threshold(0.0) == 0 and O.threshold(1.0) == 2 ** 32 and O.threshold(0.5) == 2 ** 31
    assert O.threshold(0.3) == math.floor(0.3 * 2 ** 32)


# ---------------------------------------------------------------------------
# cost model: hand values and the paper's worked example
# ---------------------------------------------------------------------------
def test_stage_cost_hand_values():
    # one device: 2e12 FLOP/s, 1e11 B/s, 10e9 B; block = 1e12 FLOP, 1e10 B streamed,
    # 4e9 B resident; head = 1e12 FLOP, 5e11 B streamed, 3e9 B resident.
    p = W.make_problem([2e12], [1e11], [10_000_000_000], [[np.inf]], [[1.0]], 4,
                       [10 ** 12], [10 ** 10], [4 * 10 ** 9], [10 ** 12], [5 * 10 ** 11],
                       [3 * 10 ** 9], [0], NP=1, ND=1)
    op = O.OracleProblem(p)
    assert op.stage_cost(0, 0, 1, 0) == 0.5          # 1e12/2e12 vs 1e10/1e11=0.1
    assert op.stage_cost(0, 0, 2, 0) == 1.0          # 2e12/2e12 vs 0.2
    assert op.stage_cost(0, 0, 3, 0) == INF          # 12e9 B > 10e9 B
    assert op.stage_cost(0, 0, 1, 1) == 5.1          # master: 2e12/2e12=1 vs 5.1e11/1e11=5.1
    assert op.stage_cost(0, 0, 2, 1) == INF          # 8e9 + 3e9 > 10e9


def test_link_cost_paper_example():
    row = [l for l in open(os.path.join(GOLDEN, "paper_worked_examples.txt")) if l.startswith("link_cost")][0]
    _, A, bits, expect = row.split()
    bw = float(bits) / 8.0  # bytes/s
    p = W.make_problem([1.0, 1.0], [1.0, 1.0], [1, 1], [[np.inf, bw], [bw, np.inf]],
                       [[1.0, 1.0], [1.0, 1.0]], 2, [1], [1], [1], [0], [0], [0], [int(A)], NP=1, ND=1)
    op = O.OracleProblem(p)
    assert op.link_cost(0, 0, 1) == pytest.approx(float(expect), rel=1e-15)


def test_link_cost_congestion_scales_bandwidth():
    p = W.make_problem([1.0, 1.0], [1.0, 1.0], [1, 1], [[np.inf, 1000.0], [1000.0, np.inf]],
                       [[1.0, 0.25], [0.25, 1.0]], 2, [1], [1], [1], [0], [0], [0], [500], NP=1, ND=1)
    assert O.OracleProblem(p).link_cost(0, 1, 0) == 2.0   # 500 B / (1000 B/s * 0.25)


# ---------------------------------------------------------------------------
# DP_Pipe against brute force
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("seed", range(40))
def test_dp_matches_brute_force(seed):
    rng = np.random.default_rng(seed)
    N = int(rng.integers(1, 11))
    M = 6
    prob = tiny_problem(rng, M, N, integer=seed % 4 != 3, head=seed % 5 != 0)
    op = O.OracleProblem(prob)
    for trial in range(4):
        m = int(rng.integers(1, M + 1))
        devs = rng.permutation(M)[:m]
        v = int(rng.integers(0, prob.V))
        got = op.dp_pipe(v, devs)
        bf = bf_dp(op, v, devs, N)
        if bf is None:
            assert not got["ok"] and got["V"] == INF and got["mu"] == -1
            continue
        V, mu, layers = bf
        assert got["ok"]
        assert got["V"] == V, (devs, v)
        assert got["mu"] == mu
        assert list(got["layers"]) == layers


def test_head_only_adds_and_a_free_head_on_device_1_decides_the_master():
    """The facts the spilled DP layout's speculation rests on (Sec. 3.2, Alg. 1),
    by enumeration: every master's optimum V_mu is at least the master-free
    optimum V0 (the head only adds cost); so when the head on device 1 leaves
    the optimum unchanged (V_1 == V0), the first-wins argmin over masters is
    device 1 and the DP's value is V0.  Small-integer costs make both cases
    (V_1 == V0 and V_1 > V0) frequent."""
    rng = np.random.default_rng(2718)
    hits = misses = 0
    for trial in range(60):
        N = int(rng.integers(2, 9))
        M = 5
        prob = tiny_problem(rng, M, N, integer=True, head=True)
        op = O.OracleProblem(prob)
        m = int(rng.integers(2, min(M, N) + 1))
        devs = rng.permutation(M)[:m]
        v = int(rng.integers(0, prob.V))
        V0 = bf_value(op, v, devs, N, m, m)                     # no device holds the head
        Vmu = [bf_value(op, v, devs, N, m, mu) for mu in range(m)]
        assert all(x >= V0 for x in Vmu), (Vmu, V0)
        if V0 == INF:
            continue
        got = op.dp_pipe(v, devs)
        if Vmu[0] == V0:
            hits += 1
            assert got["ok"] and got["mu"] == 0 and got["V"] == V0
        elif got["ok"]:
            misses += 1
            assert got["V"] == min(Vmu) >= V0
    assert hits >= 10 and misses >= 5, (hits, misses)


def test_dp_more_devices_than_blocks_is_infeasible():
    rng = np.random.default_rng(0)
    prob = tiny_problem(rng, 6, 4, tight_mem=False)
    r = O.OracleProblem(prob).dp_pipe(0, [0, 1, 2, 3, 4])
    assert not r["ok"] and r["V"] == INF and list(r["layers"]) == [-1] * 5


def test_dp_closed_form_identical_devices():
    # identical devices, free links, no head, ample memory: the optimum is the
    # cost of ceil(N/m) blocks, and the smallest-split rule puts the short
    # stages first (10 blocks on 3 devices -> 3,3,4)
    for N, m in [(10, 3), (7, 2), (12, 5), (9, 9), (1, 1), (13, 4)]:
        M = m
        p = W.make_problem(np.full(M, 3.0), np.full(M, 1.0), np.full(M, 10 ** 6),
                           np.full((M, M), np.inf), np.ones((M, M)), N, [7], [1], [1], [0], [0], [0],
                           [5], NP=1, ND=1)
        op = O.OracleProblem(p)
        r = op.dp_pipe(0, list(range(m)))
        q = math.ceil(N / m)
        assert r["V"] == (7 * q) / 3.0
        assert sum(r["layers"]) == N and max(r["layers"]) == q
        if (N, m) == (10, 3):
            assert list(r["layers"]) == [3, 3, 4]
        assert r["mu"] == 0


def test_dp_candidate_count_is_quadratic():
    # the recurrence examines N candidates for device 1 and sum_{i} (i-k+2) for
    # device k, for each of the m masters: O(m^2 N^2) as the paper states
    rng = np.random.default_rng(1)
    for N, m in [(10, 3), (20, 5), (32, 8)]:
        prob = tiny_problem(rng, 8, N, tight_mem=False)
        r = O.OracleProblem(prob).dp_pipe(0, list(range(m)))
        per_mu = N + sum((N - k + 1) * (N - k + 2) // 2 for k in range(2, m + 1))
        assert r["cand"] == m * per_mu


def _invariants(op, prob, v, devs, r):
    N = prob.N
    lay = [int(x) for x in r["layers"]]
    assert sum(lay) == N and min(lay) >= 1
    mu = r["mu"]
    worst = 0.0
    for k, d in enumerate(devs):
        c = op.stage_cost(v, int(d), lay[k], k == mu)
        assert c < INF  # memory fits
        worst = max(worst, c)
        if k:
            t = op.link_cost(v, int(devs[k - 1]), int(d))
            assert r["V"] >= t
            worst = max(worst, t)
    assert worst == r["V"]


def test_dp_invariants_on_tiny_workload():
    prob = W.make_config("c1_tiny")
    op = O.OracleProblem(prob)
    rng = np.random.default_rng(3)
    checked = 0
    for _ in range(60):
        m = int(rng.integers(1, prob.M + 1))
        devs = rng.permutation(prob.M)[:m]
        for v in (0, 1, prob.b_max):
            r = op.dp_pipe(v, devs)
            if r["ok"]:
                _invariants(op, prob, v, devs, r)
                checked += 1
                if m == 1:
                    assert r["V"] == op.stage_cost(v, int(devs[0]), prob.N, True)
    assert checked > 20


def test_dp_brute_force_on_tiny_workload_clusters():
    # real tiny-config costs, a shortened model so that enumeration stays cheap
    prob = W.make_config("c1_tiny")
    prob.N = 10
    op = O.OracleProblem(prob)
    rng = np.random.default_rng(4)
    for _ in range(12):
        m = int(rng.integers(1, 5))
        devs = rng.permutation(prob.M)[:m]
        for v in (0, prob.b_max):
            got = op.dp_pipe(v, devs)
            bf = bf_dp(op, v, devs, prob.N)
            if bf is None:
                assert not got["ok"]
            else:
                assert (got["V"], got["mu"], list(got["layers"])) == bf


# ---------------------------------------------------------------------------
# metamorphic: doubling every rate, bandwidth and link speed halves all times
# exactly (division by a power of two is exact), leaves partitions unchanged
# ---------------------------------------------------------------------------
def test_metamorphic_power_of_two_scaling():
    prob = W.make_config("c1_tiny")
    fast = W.make_config("c1_tiny")
    fast.rate = prob.rate * 2
    fast.bw = prob.bw * 2
    fast.link_bw = prob.link_bw * 2
    fast.t_a = prob.t_a / 2
    fast.min_tps = prob.min_tps * 2
    g = W.random_genomes(prob.M, prob.K_max, 48, seed=5)
    a = O.OracleProblem(prob).eval_population(g, prob.K_max)
    b = O.OracleProblem(fast).eval_population(g, prob.K_max)
    for k in ("layers", "master", "bsel"):
        assert np.array_equal(a[k], b[k])
    assert np.array_equal(a["T"] / 2, b["T"])
    assert np.array_equal(a["L"] / 2, b["L"])
    assert np.array_equal(a["fitness"][:, :2] / 2, b["fitness"][:, :2])
    assert np.array_equal(a["fitness"][:, 2:] * 2, b["fitness"][:, 2:])


# ---------------------------------------------------------------------------
# gene decoding (paper example) and the objective (Eq. 3-5)
# ---------------------------------------------------------------------------
def test_gene_decoding_paper_example():
    row = [l for l in open(os.path.join(GOLDEN, "paper_worked_examples.txt")) if l.startswith("gene")][0]
    _, body = row.split(" ", 1)
    order_s, group_s, reps_s = [x.strip() for x in body.split("|")]
    order = [int(x) for x in order_s.split(",")]
    groups = [int(x) for x in group_s.split(",")]
    reps = [[int(x) for x in r.split(",")] for r in reps_s.split(";")]
    M = len(order)
    rng = np.random.default_rng(8)
    prob = tiny_problem(rng, M, 6, tight_mem=False)
    op = O.OracleProblem(prob)
    K = 4
    sizes = np.zeros((1, K), np.uint16)
    sizes[0, :3] = groups
    g = dict(perm=np.array([order], np.uint16), sizes=sizes, nclus=np.array([3], np.uint8),
             roles=np.array([0b010], np.uint64))
    out = op.eval_population(g, K)
    off = 0
    for c, rep in enumerate(reps):
        r = op.eval_cluster(rep, decode=(c == 1))
        assert out["T"][0, c] == r["T"] and out["bsel"][0, c] == r["b"]
        assert list(out["layers"][0, off:off + len(rep)]) == list(r["layers"])
        off += len(rep)


def _objective_problem(NP, ND, t_a):
    return W.make_problem([1.0], [1.0], [1], [[np.inf]], [[1.0]], 1, [1], [1], [1], [0], [0], [0],
                          [0], NP=NP, ND=ND, t_a=t_a)


def test_objective_hand_cases():
    op = O.OracleProblem(_objective_problem(100, 100, 1.0))
    # prefill T=1 s -> PS = 100 tok/s; decode b=2 at T=0.5 s -> DS = 4 tok/s
    # Eq.3: phase = max(100/100, 100/4) = 25; Eq.4: 25 - 1 = 24; Eq.5: 1 + 24 = 25
    f = op.score(0b10, [1.0, 0.5], [0, 2])
    assert list(f) == [25.0, 25.0, 100.0, 4.0]
    # two prefill replicas aggregate (Sec. 3.3): PS = 100/1 + 100/0.5 = 300
    f = op.score(0b100, [1.0, 0.5, 0.25], [0, 0, 8])
    assert f[2] == 300.0 and f[3] == 32.0
    # phase = max(1/3, 3.125) = 3.125 -> w = 1/3 + 2.125
    assert f[1] == 3.125 and f[0] == 100.0 / 300.0 + 2.125
    # no congestion: phase below the arrival interval -> w = 0
    f = op.score(0b10, [0.01, 0.01], [0, 8])
    assert f[0] == 0.0 and f[1] == max(100 / (100 / 0.01), 100 / (8 / 0.01))
    # phase exactly T_a: bottleneck = 0, strict > in Eq. 5 -> w = 0
    f = op.score(0b10, [1.0, 0.01], [0, 1])   # PS=100 -> NP/PS = 1.0 = T_a
    assert f[1] == 1.0 and f[0] == 0.0
    # no prefill capacity, or no decode capacity -> infinite waiting
    assert op.score(0b11, [1.0, 1.0], [1, 1])[0] == INF
    assert op.score(0b00, [1.0, 1.0], [0, 0])[0] == INF
    # an infeasible replica contributes nothing
    f = op.score(0b10, [1.0, INF], [0, -1])
    assert f[0] == INF and f[2] == 100.0 and f[3] == 0.0


def test_decode_picks_highest_feasible_batch():
    prob = W.make_config("c1_tiny")
    op = O.OracleProblem(prob)
    rng = np.random.default_rng(9)
    seen_mid = 0
    for _ in range(80):
        m = int(rng.integers(1, 5))
        devs = rng.permutation(prob.M)[:m]
        r = op.eval_cluster(devs, decode=True)
        b = r["b"] if r["ok"] else 0
        for bb in range(b + 1, prob.b_max + 1):       # every larger batch fails
            d = op.dp_pipe(bb, devs)
            if d["ok"]:
                assert 1.0 / op.latency(bb, devs, d["mu"], d["layers"]) < prob.min_tps
        if r["ok"]:
            d = op.dp_pipe(b, devs)
            assert d["V"] == r["T"] and 1.0 / r["L"] >= prob.min_tps
            seen_mid += 0 < b < prob.b_max
    # the sweep must stop inside the range, not only at its ends: on these 80
    # random clusters 52 serve and 9 of them stop at a batch strictly between
    # 1 and b_max (a sweep that only tried b_max, or that stopped at the first
    # feasible batch from below, would not)
    assert seen_mid >= 5


# ---------------------------------------------------------------------------
# genetic operators
# ---------------------------------------------------------------------------
def _valid(g, M, K):
    for s in range(len(g["nclus"])):
        assert sorted(g["perm"][s]) == list(range(M))
        R = int(g["nclus"][s])
        assert 1 <= R <= min(K, M)
        sz = g["sizes"][s]
        assert all(sz[:R] >= 1) and int(sz[:R].sum()) == M and all(sz[R:] == 0)
        assert int(g["roles"][s]) >> R == 0


def test_init_population_valid_and_spread():
    ga = O._ga_struct(400, 12, 5, 13, 4, 0.5, 0.3, (0.2, 0.5, 0.15, 0.15))
    g = O.init_population(ga, 77)
    _valid(g, 12, 5)
    counts = np.bincount(g["nclus"], minlength=6)[1:]
    assert all(counts > 50)                      # R uniform over 1..5
    assert len({tuple(p) for p in g["perm"]}) > 390


def test_repair_hand_example():
    # A = 0 1 2 3 4, B = 4 3 2 1 0, B taken at positions 0 and 3 -> 4 1 2 1 4;
    # position 3 repeats 1 and position 4 repeats 4, the missing 0 and 3 fill them
    assert list(O.repair([4, 1, 2, 1, 4])) == [4, 1, 2, 0, 3]
    assert list(O.repair([2, 2, 2, 2])) == [2, 0, 1, 3]
    assert list(O.repair([3, 1, 0, 2])) == [3, 1, 0, 2]


def test_mutation_kind_frequencies():
    # kinds drawn from word 1 of the mutation stream against cumulative
    # thresholds: 20% swap, 50% regroup-from-position, 15% regroup, 15% both
    t = [O.threshold(x) for x in (0.2, 0.2 + 0.5, 0.2 + 0.5 + 0.15)]
    n = 200000
    w = np.array([O.word(11, 3, s, O.PURPOSE["MUTATE"], 1) for s in range(n)], dtype=np.uint64)
    kinds = np.searchsorted(np.array(t, dtype=np.uint64), w, side="right")
    freq = np.bincount(kinds, minlength=4) / n
    assert np.allclose(freq, [0.2, 0.5, 0.15, 0.15], atol=0.004)


def _ga_problem(P=200, M=10, K=4, Q=7, p_mut=0.3, kinds=(0.2, 0.5, 0.15, 0.15)):
    return O._ga_struct(P, M, K, Q, 4, 0.5, p_mut, kinds)


def _fitness_for(g, rng):
    P = len(g["nclus"])
    f = np.zeros((P, 4))
    f[:, 0] = rng.choice([0.0, 1.0, 2.5, INF], P)
    f[:, 1] = rng.uniform(0, 3, P)
    return f


def test_ga_children_valid_and_elites_copied():
    rng = np.random.default_rng(12)
    ga = _ga_problem()
    g = O.init_population(ga, 5)
    f = _fitness_for(g, rng)
    e = O.elites(ga, g, f)
    nxt = O.ga_step(ga, 5, 1, g, f, e)
    _valid(nxt, ga.M, ga.K)
    for q in range(ga.Q):
        for k in ("perm", "sizes"):
            assert np.array_equal(nxt[k][q], g[k][e[q]])
        assert nxt["nclus"][q] == g["nclus"][e[q]] and nxt["roles"][q] == g["roles"][e[q]]


def test_ga_mutation_kinds_act_as_described():
    rng = np.random.default_rng(13)
    base = _ga_problem(p_mut=0.0)
    g = O.init_population(base, 9)
    f = _fitness_for(g, rng)
    e = O.elites(base, g, f)
    plain = O.ga_step(base, 9, 2, g, f, e)       # crossover + repair only
    Q = base.Q
    # swap only: the ordering differs from the unmutated child by one transposition
    sw = O.ga_step(_ga_problem(p_mut=1.0, kinds=(1.0, 0, 0, 0)), 9, 2, g, f, e)
    for s in range(Q, base.P):
        diff = np.nonzero(sw["perm"][s] != plain["perm"][s])[0]
        assert len(diff) in (0, 2)
        assert np.array_equal(sw["sizes"][s], plain["sizes"][s])
    # regroup from a position: ordering untouched, a prefix of the grouping kept
    rg = O.ga_step(_ga_problem(p_mut=1.0, kinds=(0, 1.0, 0, 0)), 9, 2, g, f, e)
    _valid(rg, base.M, base.K)
    for s in range(Q, base.P):
        assert np.array_equal(rg["perm"][s], plain["perm"][s])
    # regenerate both: orderings change (almost surely)
    bo = O.ga_step(_ga_problem(p_mut=1.0, kinds=(0, 0, 0, 1.0)), 9, 2, g, f, e)
    _valid(bo, base.M, base.K)
    changed = sum(not np.array_equal(bo["perm"][s], plain["perm"][s]) for s in range(Q, base.P))
    assert changed > (base.P - Q) * 0.9


def _distinct_population(P, M, K, seed):
    """P genomes with pairwise distinct orderings (so that an ordering names
    its genome) and at least two replicas each; drawn by numpy."""
    rng = np.random.default_rng(seed)
    perms = set()
    g = O.empty_genomes(P, M, K)
    s = 0
    while s < P:
        perm = tuple(int(x) for x in rng.permutation(M))
        R = int(rng.integers(2, K + 1))
        cuts = tuple(sorted(int(x) for x in rng.choice(np.arange(1, M), R - 1, replace=False)))
        if perm in perms:
            continue
        perms.add(perm)
        edges = (0,) + cuts + (M,)
        g["perm"][s] = perm
        g["sizes"][s, :R] = np.diff(edges)
        g["nclus"][s] = R
        g["roles"][s] = int(rng.integers(0, 1 << R))
        s += 1
    return g


def _same_genome(a, i, b, j):
    return all(np.array_equal(a[k][i], b[k][j]) for k in ("perm", "sizes", "nclus", "roles"))


def test_tournament_keeps_the_fittest():
    # App. A selects parents "based on fitness": a tournament returns its best
    # entrant.  One genome is strictly best; with 256 entrants per tournament
    # over 16 genomes it is drawn with probability 1 - (15/16)^256 > 1 - 1e-7,
    # so with no mutation both parents of every child are that genome and the
    # child equals it (crossover of two copies, repair a no-op).  Keeping the
    # worst entrant instead would clone the worst genome.
    P, M, K = 16, 9, 4
    g = _distinct_population(P, M, K, 31)
    f = np.zeros((P, 4))
    f[:, 0] = np.arange(P, 0, -1, dtype=float)      # genome P-1 is the best (w = 1)
    best = P - 1
    ga = O._ga_struct(P, M, K, 0, 256, 0.5, 0.0, (0.2, 0.5, 0.15, 0.15))
    nxt = O.ga_step(ga, 4, 1, g, f, np.zeros(0, np.int32))
    for s in range(P):
        assert _same_genome(nxt, s, g, best)
    # ties on w are broken by the bottleneck phase, then by the lower index
    f[:, 0] = 1.0
    f[:, 1] = 2.0
    f[5, 1] = 1.5
    nxt = O.ga_step(ga, 4, 1, g, f, np.zeros(0, np.int32))
    assert all(_same_genome(nxt, s, g, 5) for s in range(P))
    f[:, 1] = 2.0
    nxt = O.ga_step(ga, 4, 1, g, f, np.zeros(0, np.int32))
    assert all(_same_genome(nxt, s, g, 0) for s in range(P))


def test_grouping_comes_whole_from_either_parent():
    # Sec. 3.4: crossover recombines the ordering and inherits the grouping
    # chromosome from one parent.  With p_cx = 0 the child's ordering is parent
    # A's, with p_cx = 1 parent B's (the parent draws do not depend on p_cx), so
    # the two runs name both parents of every child; the grouping and roles
    # must then be A's or B's whole, and over many children each parent gives
    # it about half the time (a fair coin).
    P, M, K = 600, 12, 5
    g = _distinct_population(P, M, K, 32)
    rng = np.random.default_rng(33)
    f = np.zeros((P, 4))
    f[:, 0] = rng.permutation(P).astype(float)
    order_of = {tuple(g["perm"][i]): i for i in range(P)}
    ga0 = O._ga_struct(P, M, K, 0, 2, 0.0, 0.0, (0.2, 0.5, 0.15, 0.15))
    ga1 = O._ga_struct(P, M, K, 0, 2, 1.0, 0.0, (0.2, 0.5, 0.15, 0.15))
    none = np.zeros(0, np.int32)
    a_run = O.ga_step(ga0, 8, 3, g, f, none)
    b_run = O.ga_step(ga1, 8, 3, g, f, none)
    from_b = both = 0
    for s in range(P):
        A = order_of[tuple(a_run["perm"][s])]
        B = order_of[tuple(b_run["perm"][s])]
        for run in (a_run, b_run):
            src = [x for x in (A, B) if np.array_equal(run["sizes"][s], g["sizes"][x])
                   and run["nclus"][s] == g["nclus"][x] and run["roles"][s] == g["roles"][x]]
            assert src, "grouping and roles must come whole from a parent"
        # the same coin in both runs: the grouping source does not depend on p_cx
        assert np.array_equal(a_run["sizes"][s], b_run["sizes"][s])
        if not np.array_equal(g["sizes"][A], g["sizes"][B]):
            both += 1
            from_b += np.array_equal(a_run["sizes"][s], g["sizes"][B])
    assert both > 450
    assert 0.42 < from_b / both < 0.58


def test_regroup_from_a_position_keeps_the_prefix():
    # App. A: "regenerates the grouping from a random position".  The replica r
    # is uniform over the source's R replicas (word 2 of the mutation stream);
    # replicas [0, r) keep their sizes and roles, the ordering is untouched, and
    # the devices from replica r on are regrouped.  Most children (all with
    # r >= 1) therefore keep a non-empty prefix.
    P, M, K = 400, 40, 8
    g = _distinct_population(P, M, K, 34)
    rng = np.random.default_rng(35)
    f = np.zeros((P, 4))
    f[:, 0] = rng.permutation(P).astype(float)
    none = np.zeros(0, np.int32)
    plain = O.ga_step(O._ga_struct(P, M, K, 0, 4, 0.5, 0.0, (0.2, 0.5, 0.15, 0.15)), 6, 2, g, f, none)
    rg = O.ga_step(O._ga_struct(P, M, K, 0, 4, 0.5, 1.0, (0.0, 1.0, 0.0, 0.0)), 6, 2, g, f, none)
    _valid(rg, M, K)
    kept_some = 0
    for s in range(P):
        assert np.array_equal(rg["perm"][s], plain["perm"][s])
        R = int(plain["nclus"][s])
        r = (O.word(6, 2, s, O.PURPOSE["MUTATE"], 2) * R) >> 32
        assert np.array_equal(rg["sizes"][s][:r], plain["sizes"][s][:r])
        mask = (1 << r) - 1
        assert int(rg["roles"][s]) & mask == int(plain["roles"][s]) & mask
        assert int(rg["nclus"][s]) >= r + 1
        kept_some += r >= 1
    # R >= 2 for every source, so r >= 1 for at least half of the children
    assert kept_some > 0.5 * P


def test_regroup_all_keeps_the_ordering():
    # App. A's third mutation kind regenerates the grouping entirely and leaves
    # the ordering as crossover made it; the fourth regenerates both.  With
    # every mutation of the third kind, no ordering changes and (almost) every
    # grouping does.
    P, M, K = 300, 20, 6
    g = _distinct_population(P, M, K, 36)
    rng = np.random.default_rng(37)
    f = np.zeros((P, 4))
    f[:, 0] = rng.permutation(P).astype(float)
    none = np.zeros(0, np.int32)
    plain = O.ga_step(O._ga_struct(P, M, K, 0, 4, 0.5, 0.0, (0.2, 0.5, 0.15, 0.15)), 7, 5, g, f, none)
    ra = O.ga_step(O._ga_struct(P, M, K, 0, 4, 0.5, 1.0, (0.0, 0.0, 1.0, 0.0)), 7, 5, g, f, none)
    _valid(ra, M, K)
    changed = 0
    for s in range(P):
        assert np.array_equal(ra["perm"][s], plain["perm"][s])
        changed += not (np.array_equal(ra["sizes"][s], plain["sizes"][s]) and ra["roles"][s] == plain["roles"][s])
    assert changed > 0.9 * P
    # and the kind boundaries sit at the cumulative 0.2 / 0.7 / 0.85: with the
    # paper's mix, a child mutated with a kind word in [0.7, 0.85) keeps its
    # ordering, one with a word at or above 0.85 gets a new one
    mix = O.ga_step(O._ga_struct(P, M, K, 0, 4, 0.5, 1.0, (0.2, 0.5, 0.15, 0.15)), 7, 5, g, f, none)
    t2, t3 = O.threshold(0.7), O.threshold(0.85)
    n3 = n4 = 0
    for s in range(P):
        kw = O.word(7, 5, s, O.PURPOSE["MUTATE"], 1)
        if t2 <= kw < t3:
            n3 += 1
            assert np.array_equal(mix["perm"][s], plain["perm"][s])
        elif kw >= t3:
            n4 += not np.array_equal(mix["perm"][s], plain["perm"][s])
    assert n3 > 20 and n4 > 20


def test_crossover_mixes_both_parents_evenly():
    # with identical fitness everywhere the tournament picks by index; check the
    # per-position source statistics of a uniform crossover at p = 0.5
    n = 100000
    w = np.array([O.word(21, 1, s, O.PURPOSE["CROSS"], 3) for s in range(n)], dtype=np.uint64)
    assert abs(np.mean(w < O.threshold(0.5)) - 0.5) < 0.005


def test_elites_distinct_and_ordered():
    ga = _ga_problem(P=12, M=5, K=3, Q=6)
    g = O.init_population(ga, 3)
    # make genomes 4 and 9 copies of genome 1, genome 7 a copy of 2
    for dst, src in [(4, 1), (9, 1), (7, 2)]:
        for k in ("perm", "sizes", "nclus", "roles"):
            g[k][dst] = g[k][src]
    f = np.zeros((12, 4))
    f[:, 0] = [5, 1, 2, 9, 1, 0.5, 7, 2, 8, 1, 3, 4]
    f[:, 1] = 0
    e = list(O.elites(ga, g, f))
    # distinct genomes by (w, index): 5(0.5) 1(1) 2(2) 10(3) 11(4) 0(5)
    assert e == [5, 1, 2, 10, 11, 0]
    ga2 = _ga_problem(P=12, M=5, K=3, Q=11)
    e2 = list(O.elites(ga2, g, f))
    # 9 distinct genomes, then duplicates by key: 4 (w=1), 9 (w=1)
    assert e2 == [5, 1, 2, 10, 11, 0, 6, 8, 3, 4, 9]


def test_ga_best_is_monotone_and_bounded_by_exhaustive_optimum():
    # 5 devices, at most 2 replicas: enumerate every genome for the optimum
    rng = np.random.default_rng(21)
    M, K, N = 5, 2, 6
    prob = tiny_problem(rng, M, N, integer=False, tight_mem=False)
    prob.t_a = 0.0
    op = O.OracleProblem(prob)
    allg = []
    for perm in itertools.permutations(range(M)):
        for R in (1, 2):
            for comp in compositions(M, R):
                for roles in range(1 << R):
                    allg.append((perm, comp, R, roles))
    P_all = len(allg)
    G = dict(perm=np.array([a[0] for a in allg], np.uint16),
             sizes=np.array([list(a[1]) + [0] * (K - a[2]) for a in allg], np.uint16),
             nclus=np.array([a[2] for a in allg], np.uint8),
             roles=np.array([a[3] for a in allg], np.uint64))
    opt = op.eval_population(G, K, nthreads=4)["fitness"][:, 0].min()
    ga = O._ga_struct(32, M, K, 2, 4, 0.5, 0.3, (0.2, 0.5, 0.15, 0.15))
    g = O.init_population(ga, 1)
    best = INF
    for gen in range(1, 12):
        f = op.eval_population(g, K)["fitness"]
        cur = f[:, 0].min()
        assert cur >= opt
        assert cur <= best
        best = cur
        e = O.elites(ga, g, f)
        g = O.ga_step(ga, 1, gen, g, f, e)
    assert P_all == 120 * (2 + 4 * 4)


def test_congestion_redraw_range_and_symmetry():
    c = O.redraw_congestion(64, 3, 5, 0.2, 1.0)
    off = c[~np.eye(64, dtype=bool)]
    assert np.array_equal(c, c.T) and np.all(np.diag(c) == 1.0)
    assert off.min() >= 0.2 and off.max() < 1.0
    assert abs(off.mean() - 0.6) < 0.01
    c2 = O.redraw_congestion(64, 3, 6, 0.2, 1.0)
    assert not np.array_equal(c, c2)
    assert np.array_equal(c, O.redraw_congestion(64, 3, 5, 0.2, 1.0))


def test_memory_boundary_fits_exactly():
    # a stage that needs exactly the device's memory fits (infeasible only if it exceeds)
    p = W.make_problem([1.0], [1.0], [12], [[np.inf]], [[1.0]], 4, [1], [1], [4], [0], [0], [4],
                       [0], NP=1, ND=1)
    op = O.OracleProblem(p)
    assert op.stage_cost(0, 0, 3, 0) == 3.0
    assert op.stage_cost(0, 0, 2, 1) == 2.0     # 2*4 + 4 = 12 bytes = memory
    assert op.stage_cost(0, 0, 3, 1) == INF


def test_latency_hand_value_and_tps_boundary():
    # decode b=1: a block is 1 FLOP on 4 FLOP/s devices (0.25 s), the activation
    # 1 byte over a 4 B/s link (0.25 s): two devices, one block each ->
    # Lambda = 0.25 + 0.25 + 0.25 = 0.75 s, bottleneck T = 0.25 s.
    # Sec. 3.2: a per-request rate 1/Lambda that equals Min_TPS is accepted.
    link = [[np.inf, 4.0], [4.0, np.inf]]
    mk = lambda tps: W.make_problem([4.0, 4.0], [1.0, 1.0], [10, 10], link, np.ones((2, 2)), 2,
                                    [1, 1], [0, 0], [1, 1], [0, 0], [0, 0], [0, 0], [1, 1],
                                    NP=1, ND=1, min_tps=tps)
    op = O.OracleProblem(mk(1.0 / 0.75))
    d = op.dp_pipe(1, [0, 1])
    assert d["V"] == 0.25 and list(d["layers"]) == [1, 1]
    assert op.latency(1, [0, 1], d["mu"], d["layers"]) == 0.75
    r = op.eval_cluster([0, 1], decode=True)
    assert r["ok"] and r["b"] == 1 and r["T"] == 0.25 and r["L"] == 0.75
    r = O.OracleProblem(mk(np.nextafter(1.0 / 0.75, 2.0))).eval_cluster([0, 1], decode=True)
    assert not r["ok"] and r["b"] == -1


def test_role_search_is_the_best_fixed_assignment():
    """Alg. 2's role search: the fitness equals the least (w, phase) over every
    role assignment evaluated with fixed role bits, the smallest such
    assignment is chosen, the replicas' outputs are those of that assignment,
    and the genome's own role bits do not matter."""
    import dataclasses
    prob = W.make_config("c1_tiny")
    search = O.OracleProblem(dataclasses.replace(prob, role_search=1))
    fixed = O.OracleProblem(prob)
    K = 5
    g = W.random_genomes(prob.M, K, 24, seed=31)
    got = search.eval_population(g, K)
    scrambled = dict(g, roles=np.ascontiguousarray(g["roles"] ^ np.uint64(0b10110)))
    again = search.eval_population(scrambled, K)
    for key in ("fitness", "layers", "master", "bsel", "T", "L", "roles"):
        assert np.array_equal(got[key], again[key]), key
    checked_feasible = 0
    for p in range(24):
        R = int(g["nclus"][p])
        one = {k: np.repeat(v[p:p + 1], 1 << R, axis=0) for k, v in g.items()}
        one["roles"] = np.arange(1 << R, dtype=np.uint64)
        every = fixed.eval_population(one, K)
        f = every["fitness"]
        best = min(range(1 << R), key=lambda r: (f[r, 0], f[r, 1], r))
        assert int(got["roles"][p]) == best
        assert np.array_equal(got["fitness"][p], f[best])
        for key in ("layers", "master", "bsel", "T", "L"):
            assert np.array_equal(got[key][p], every[key][best]), key
        checked_feasible += bool(np.isfinite(f[best, 0]))
    assert checked_feasible >= 10


# ---------------------------------------------------------------------------
# comparison objectives (Sec. 4.2 "Baseline chosen")
# ---------------------------------------------------------------------------
def _ft_problem(NP, ND):
    import dataclasses
    return dataclasses.replace(_objective_problem(NP, ND, 1.0), objective=1)


def test_finishing_time_hand_cases():
    """HexGen-2's per-request finishing time: a request's prefill pass plus ND
    decode passes, each the end-to-end latency Lambda of its replica (stages
    and links added), averaged over the replicas of a role in proportion to
    their rates."""
    op = O.OracleProblem(_ft_problem(100, 50))
    # one replica per role: FT = Lambda_P + ND * Lambda_D = 5 + 50 * 3
    f = op.score(0b10, [2.0, 0.5], [0, 4], L=[5.0, 3.0])
    assert f[0] == 155.0
    assert f[2] == 50.0 and f[3] == 8.0 and f[1] == max(100 / 50, 50 / 8)   # PS, DS and Eq. 3 unchanged
    # two equally fast prefill replicas with latencies 2 and 6: their mean, 4
    f = op.score(0b100, [1.0, 1.0, 1.0], [0, 0, 1], L=[2.0, 6.0, 1.0])
    assert f[0] == 4.0 + 50 * 1.0
    # rate-weighted: prefill rates 3 and 1 tok/s (NP = 3, T = 1 and 3), latencies
    # 1 and 3 -> (3*1 + 1*3) / 4 = 1.5
    op3 = O.OracleProblem(_ft_problem(3, 1))
    f = op3.score(0b100, [1.0, 3.0, 1.0], [0, 0, 1], L=[1.0, 3.0, 2.0])
    assert f[0] == 1.5 + 1 * 2.0
    # the waiting-time objective on the same replicas ignores Lambda
    assert O.OracleProblem(_objective_problem(3, 1, 1.0)).score(0b100, [1.0, 3.0, 1.0], [0, 0, 1],
                                                                L=[1.0, 3.0, 2.0])[0] == 0.0
    # no decode capacity, or an infeasible replica alone in its role: +inf
    assert op.score(0b00, [1.0, 1.0], [0, 0], L=[1.0, 1.0])[0] == INF
    assert op.score(0b10, [1.0, INF], [0, -1], L=[1.0, INF])[0] == INF


def test_finishing_time_scales_with_time():
    """Every rate, bandwidth and link speed doubled: every stage and link time
    halves exactly, and so does FT (a sum of latencies; ND is a count)."""
    import dataclasses
    prob = dataclasses.replace(W.make_config("c1_tiny"), objective=1)
    fast = dataclasses.replace(prob, rate=prob.rate * 2, bw=prob.bw * 2, link_bw=prob.link_bw * 2,
                               min_tps=prob.min_tps * 2)
    g = W.random_genomes(prob.M, prob.K_max, 240, seed=41)
    a = O.OracleProblem(prob).eval_population(g, prob.K_max)
    b = O.OracleProblem(fast).eval_population(g, prob.K_max)
    fin = np.isfinite(a["fitness"][:, 0])
    assert fin.sum() >= 20
    assert np.array_equal(a["fitness"][:, 0] / 2, b["fitness"][:, 0])
    assert np.array_equal(a["layers"], b["layers"]) and np.array_equal(a["bsel"], b["bsel"])


def test_finishing_time_role_search_is_the_best_fixed_assignment():
    import dataclasses
    prob = dataclasses.replace(W.make_config("c1_tiny"), objective=1)
    search = O.OracleProblem(dataclasses.replace(prob, role_search=1))
    fixed = O.OracleProblem(prob)
    K = 4
    g = W.random_genomes(prob.M, K, 16, seed=43)
    got = search.eval_population(g, K)
    finite = 0
    for p in range(16):
        R = int(g["nclus"][p])
        one = {k: np.repeat(v[p:p + 1], 1 << R, axis=0) for k, v in g.items()}
        one["roles"] = np.arange(1 << R, dtype=np.uint64)
        f = fixed.eval_population(one, K)["fitness"]
        best = min(range(1 << R), key=lambda r: (f[r, 0], f[r, 1], r))
        assert int(got["roles"][p]) == best and np.array_equal(got["fitness"][p], f[best])
        finite += bool(np.isfinite(f[best, 0]))
    assert finite >= 6


def test_splitwise_prefill_count():
    """SplitWise sizes its pools by the input-to-generated token ratio: R
    replicas split NP : ND, rounded half up, at least one per role."""
    cases = {(1, 1, 4): 2, (1, 1, 1): 1, (1, 1, 2): 1, (3, 1, 4): 3, (1, 3, 4): 1, (1, 1, 3): 2,
             (1, 100, 3): 1, (100, 1, 3): 2, (2291, 1385, 10): 6, (576, 746, 10): 4, (5, 5, 64): 32}
    for (NP, ND, R), n in cases.items():
        assert O.splitwise_prefill_count(NP, ND, R) == n, (NP, ND, R)


def _single_device_replicas(rates, NP=64, ND=64):
    """Replicas of one device each, identical but for the compute rate, with
    ample memory and free links: the prefill throughput orders as the rate."""
    M = len(rates)
    V = 3
    return W.make_problem(rates, [1e12] * M, [10 ** 12] * M, np.full((M, M), np.inf), np.ones((M, M)), 4,
                          [1000] * V, [10] * V, [1] * V, [0] * V, [0] * V, [0] * V, [16] * V, NP=NP, ND=ND,
                          min_tps=0.0, role_search=2)


def test_splitwise_strongest_replicas_prefill():
    prob = _single_device_replicas([1e6, 4e6, 2e6, 3e6])
    op = O.OracleProblem(prob)
    g = dict(perm=np.array([[0, 1, 2, 3]], np.uint16), sizes=np.array([[1, 1, 1, 1]], np.uint16),
             nclus=np.array([4], np.uint8), roles=np.array([0b1111], np.uint64))
    out = op.eval_population(g, 4)
    # the two strongest (rates 4e6 and 3e6, replicas 1 and 3) prefill; 0 and 2 decode
    assert int(out["roles"][0]) == 0b0101
    assert list(out["bsel"][0]) == [2, 0, 2, 0]
    # equal strengths: the lower index prefills first
    op2 = O.OracleProblem(_single_device_replicas([2e6, 2e6, 2e6, 2e6]))
    assert int(op2.eval_population(g, 4)["roles"][0]) == 0b1100
    # NP : ND = 3 : 1 -> three prefill replicas
    op3 = O.OracleProblem(_single_device_replicas([1e6, 4e6, 2e6, 3e6], NP=96, ND=32))
    assert int(op3.eval_population(g, 4)["roles"][0]) == 0b0001


def test_splitwise_never_beats_the_role_search():
    """The adapted-SplitWise rule picks one of the 2^R assignments, so its
    (w, phase) is never below Alg. 2's brute force; its fitness is the
    objective of the assignment it picked, and its prefill replicas are at
    least as strong as its decode replicas."""
    import dataclasses
    for objective in (0, 1):
        prob = dataclasses.replace(W.make_config("c1_tiny"), objective=objective)
        K = 5
        g = W.random_genomes(prob.M, K, 40, seed=47 + objective)
        spw = O.OracleProblem(dataclasses.replace(prob, role_search=2)).eval_population(g, K)
        bf = O.OracleProblem(dataclasses.replace(prob, role_search=1)).eval_population(g, K)
        fixed = O.OracleProblem(prob).eval_population(dict(g, roles=spw["roles"]), K)
        assert np.array_equal(fixed["fitness"], spw["fitness"])
        worse = 0
        for p in range(40):
            a, b = spw["fitness"][p], bf["fitness"][p]
            assert (a[0], a[1]) >= (b[0], b[1])
            worse += (a[0], a[1]) > (b[0], b[1])
        assert worse >= 1


# ---------------------------------------------------------------------------
# GPU-CPU offload in the cost model (Sec. 1; the plans' G--C column, Sec. 4.3)
# ---------------------------------------------------------------------------
def _with_host(prob, rng, integer=True):
    """Give every other device host memory for a few blocks and a slower host."""
    import dataclasses
    M = prob.M
    mem_cpu = np.where(np.arange(M) % 2 == 0, rng.integers(1, 8, M), 0).astype(np.uint64)
    if integer:
        rate_cpu = rng.choice([0.25, 0.5], M)
        bw_cpu = rng.choice([0.5, 1.0], M)
    else:
        rate_cpu = rng.uniform(0.1, 0.5, M)
        bw_cpu = rng.uniform(0.1, 0.5, M)
    return dataclasses.replace(prob, rate_cpu=rate_cpu, bw_cpu=bw_cpu, mem_cpu=mem_cpu)


def test_offload_stage_cost_hand_values():
    # device: 2 FLOP/s, 4 B/s, 7 B; block: 2 FLOP, 4 B, 2 B resident; head: 1, 1, 1
    # host: 1 FLOP/s, 1 B/s, 5 B (two blocks)
    prob = W.make_problem([2.0], [4.0], [7], [[np.inf]], [[1.0]], 8, [2], [4], [2], [1], [1], [1], [0],
                          NP=1, ND=1, rate_cpu=[1.0], bw_cpu=[1.0], mem_cpu=[5])
    op = O.OracleProblem(prob)
    # 3 blocks fit in device memory: max(6/2, 12/4) = 3
    assert op.stage_cost(0, 0, 3, False) == 3.0 and op.gpu_blocks(0, 0, 3, False) == 3
    # 5 blocks: 3 on the device (3 s) + 2 on the host, max(4/1, 8/1) = 8 s
    assert op.stage_cost(0, 0, 5, False) == 11.0 and op.gpu_blocks(0, 0, 5, False) == 3
    # as master: the head takes 1 B of device memory (still 3 blocks fit):
    # max(7/2, 13/4) = 3.5, plus 8 on the host
    assert op.stage_cost(0, 0, 5, True) == 11.5 and op.gpu_blocks(0, 0, 5, True) == 3
    # 6 blocks: 3 offloaded need 6 B of host memory, 5 available -> infeasible
    assert op.stage_cost(0, 0, 6, False) == INF
    # no host memory: the base model (5 blocks need 10 B > 7 B)
    import dataclasses
    base = O.OracleProblem(dataclasses.replace(prob, mem_cpu=np.zeros(1, np.uint64)))
    assert base.stage_cost(0, 0, 5, False) == INF and base.stage_cost(0, 0, 3, False) == 3.0
    # a head that does not fit in device memory cannot be placed at all
    big = O.OracleProblem(dataclasses.replace(prob, head_mem=np.array([8], np.uint64)))
    assert big.stage_cost(0, 0, 1, True) == INF and big.stage_cost(0, 0, 1, False) == 1.0


def test_offload_plan_column_example():
    """The form of the plans' G--C column: a master with device memory for 20
    of a 24-block model's blocks beside the head runs 20--4 with the rest in
    host memory; with more KV slots per block (a larger decode batch) fewer
    blocks fit on the device (the decode replicas' splits shift toward the
    host)."""
    bm = [100, 115]                          # block bytes resident: prefill, decode with more slots
    prob = W.make_problem([1e12], [1e11], [20 * 100 + 50 + 99], [[np.inf]], [[1.0]], 24, [10, 10], [10, 10], bm,
                          [5, 5], [5, 5], [50, 50], [0, 0], NP=1, ND=1, rate_cpu=[1e11], bw_cpu=[1e10],
                          mem_cpu=[10 ** 6])
    op = O.OracleProblem(prob)
    assert op.gpu_blocks(0, 0, 24, True) == 20          # 20--4
    assert op.gpu_blocks(1, 0, 24, True) == 18          # 18--6
    assert op.stage_cost(0, 0, 24, True) < INF


def test_offload_without_host_memory_is_the_base_model():
    import dataclasses
    for name in ("c1_tiny", "c2"):
        prob = W.make_config(name, P=64)
        host = W.make_config(name, P=64, offload=True)
        none = dataclasses.replace(host, mem_cpu=np.zeros(prob.M, np.uint64))
        g = W.random_genomes(prob.M, prob.K_max, 64, seed=3)
        a = O.OracleProblem(prob).eval_population(g, prob.K_max, nthreads=4)
        b = O.OracleProblem(none).eval_population(g, prob.K_max, nthreads=4)
        for k in ("fitness", "layers", "master", "bsel", "T", "L"):
            assert np.array_equal(a[k], b[k]), (name, k)
        # the fleet's own draws do not move when the host side is drawn
        for k in ("rate", "bw", "mem", "link_bw", "cong"):
            assert np.array_equal(getattr(prob, k), getattr(host, k))


def test_offload_device_first_split_is_the_fastest():
    """With the host slower per block than the device, filling device memory
    first is the fastest of all feasible device/host splits of a stage."""
    rng = np.random.default_rng(61)
    for _ in range(30):
        prob = _with_host(tiny_problem(rng, 4, 9, V=3, integer=False), rng, integer=False)
        op = O.OracleProblem(prob)
        for d in range(4):
            for v in range(3):
                for n in range(1, 10):
                    for master in (False, True):
                        got = op.stage_cost(v, d, n, master)
                        hm = int(prob.head_mem[v]) if master else 0
                        bm = int(prob.blk_mem[v])
                        best = INF
                        for g in range(0, n + 1):
                            c = n - g
                            if g * bm + hm > int(prob.mem[d]) or c * bm > int(prob.mem_cpu[d]):
                                continue
                            fl = g * int(prob.blk_flops[v]) + (int(prob.head_flops[v]) if master else 0)
                            by = g * int(prob.blk_bytes[v]) + (int(prob.head_bytes[v]) if master else 0)
                            t = max(fl / prob.rate[d], by / prob.bw[d])
                            if c:
                                t += max(c * int(prob.blk_flops[v]) / prob.rate_cpu[d],
                                         c * int(prob.blk_bytes[v]) / prob.bw_cpu[d])
                            best = min(best, t)
                        per_dev = max(int(prob.blk_flops[v]) / prob.rate[d], int(prob.blk_bytes[v]) / prob.bw[d])
                        per_host = max(int(prob.blk_flops[v]) / prob.rate_cpu[d],
                                       int(prob.blk_bytes[v]) / prob.bw_cpu[d])
                        if per_host >= per_dev:
                            assert got == best or (got == INF and best == INF) or abs(got - best) <= 1e-12 * best


@pytest.mark.parametrize("seed", range(16))
def test_offload_dp_matches_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    N = int(rng.integers(1, 11))
    M = 6
    prob = _with_host(tiny_problem(rng, M, N, integer=seed % 4 != 3, head=seed % 5 != 0), rng,
                      integer=seed % 4 != 3)
    op = O.OracleProblem(prob)
    for trial in range(4):
        m = int(rng.integers(1, M + 1))
        devs = rng.permutation(M)[:m]
        v = int(rng.integers(0, prob.V))
        got = op.dp_pipe(v, devs)
        bf = bf_dp(op, v, devs, N)
        if bf is None:
            assert not got["ok"]
            continue
        V, mu, layers = bf
        assert got["ok"] and got["V"] == V and got["mu"] == mu and list(got["layers"]) == layers


def test_offload_metamorphic_power_of_two_scaling():
    prob = W.make_config("c1_tiny", offload=True)
    import dataclasses
    fast = dataclasses.replace(prob, rate=prob.rate * 2, bw=prob.bw * 2, link_bw=prob.link_bw * 2,
                               rate_cpu=prob.rate_cpu * 2, bw_cpu=prob.bw_cpu * 2, t_a=prob.t_a / 2,
                               min_tps=prob.min_tps * 2)
    g = W.random_genomes(prob.M, prob.K_max, 64, seed=8)
    a = O.OracleProblem(prob).eval_population(g, prob.K_max)
    b = O.OracleProblem(fast).eval_population(g, prob.K_max)
    for k in ("layers", "master", "bsel"):
        assert np.array_equal(a[k], b[k])
    assert np.array_equal(a["T"] / 2, b["T"]) and np.array_equal(a["L"] / 2, b["L"])
    assert np.array_equal(a["fitness"][:, :2] / 2, b["fitness"][:, :2])
    # offloading changes plans: more replicas serve than without host memory
    base = O.OracleProblem(W.make_config("c1_tiny")).eval_population(g, prob.K_max)
    assert (a["bsel"] >= 0).sum() > (base["bsel"] >= 0).sum()


# ---------------------------------------------------------------------------
# Alg. 2's role search beyond 20 replicas: only replicas that can decode vary
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("objective,t_a", [(0, 1.0), (0, 1e4), (1, 1.0)])
def test_role_search_matches_the_plain_enumeration(objective, t_a):
    """The search enumerates the roles of the replicas that can decode only (a
    replica that cannot decode prefills in the winning assignment).  Against
    the plain enumeration of all 2^R masks (R <= 14): tie-heavy small-integer
    fleets, the w = 0 plateau (a large T_a), the finishing time, and the
    128-device workload's fleet at up to 14 replicas."""
    import dataclasses
    rng = np.random.default_rng(71 + objective + int(t_a))
    cases = []
    for _ in range(3):
        M, N = 16, 10
        prob = tiny_problem(rng, M, N, V=3, integer=True)
        prob = dataclasses.replace(prob, min_tps=0.02, t_a=t_a, objective=objective)
        cases.append((prob, W.random_genomes(M, 14, 10, seed=int(rng.integers(1 << 30)), max_clusters=14), 14))
    c3 = dataclasses.replace(W.make_config("c3"), t_a=t_a, objective=objective)
    cases.append((c3, W.random_genomes(c3.M, 14, 6, seed=5, max_clusters=14), 14))
    seen_free = seen_forced = 0
    for prob, g, K in cases:
        fast = O.OracleProblem(dataclasses.replace(prob, role_search=1)).eval_population(g, K, nthreads=4)
        full = O.OracleProblem(dataclasses.replace(prob, role_search=3)).eval_population(g, K, nthreads=4)
        for k in ("fitness", "layers", "master", "bsel", "T", "L", "roles"):
            assert np.array_equal(fast[k], full[k]), k
        assert fast["capped"] == 0
        dec = O.OracleProblem(dataclasses.replace(prob, role_search=0))
        for p in range(len(g["nclus"])):
            off = 0
            for c in range(int(g["nclus"][p])):
                m = int(g["sizes"][p, c])
                can = m <= prob.N and dec.eval_cluster(g["perm"][p, off:off + m], decode=True)["ok"]
                off += m
                if objective == 1:
                    can = can or (m <= prob.N and dec.eval_cluster(g["perm"][p, off - m:off], decode=False)["ok"])
                if not can:
                    assert (int(fast["roles"][p]) >> c) & 1 == 0       # forced to prefill
                    seen_forced += 1
                else:
                    seen_free += 1
    assert seen_free >= 20 and seen_forced >= 20


def test_role_search_caps_at_twenty_decoding_replicas():
    """More than 20 replicas that can decode: the search is not run; the
    replicas keep the genome's own role bits (those that cannot decode
    prefill), and the genome is counted as capped."""
    import dataclasses
    M = 24
    prob = dataclasses.replace(_single_device_replicas([1e6 * (1 + i % 5) for i in range(M)]), role_search=1)
    K = M
    g = dict(perm=np.arange(M, dtype=np.uint16)[None, :].copy(), sizes=np.ones((1, K), np.uint16),
             nclus=np.array([M], np.uint8), roles=np.array([0b1010_1100_0011_0101_1100_1010], np.uint64))
    out = O.OracleProblem(prob).eval_population(g, K)
    assert out["capped"] == 1 and int(out["roles"][0]) == int(g["roles"][0])
    fixed = O.OracleProblem(dataclasses.replace(prob, role_search=0)).eval_population(g, K)
    assert np.array_equal(out["fitness"], fixed["fitness"])
    # 20 decoding replicas (4 more that cannot serve at all): the search runs
    prob20 = dataclasses.replace(prob, mem=np.array([10 ** 12] * 20 + [0] * 4, np.uint64))
    out20 = O.OracleProblem(prob20).eval_population(g, K)
    assert out20["capped"] == 0 and int(out20["roles"][0]) >> 20 == 0


# ---------------------------------------------------------------------------
# blocks of several types: per-layer prefix sums PF, PB, PM (Sec. 3.1)
# ---------------------------------------------------------------------------
def _layered(prob, rng, integer=True):
    """Per-layer work for a tiny problem: block l's flops, bytes and resident
    bytes drawn per variant (small integers: heavy and light blocks, ties)."""
    import dataclasses
    V, N = prob.V, prob.N
    f = rng.integers(1, 6, (V, N)) if integer else rng.integers(1, 1000, (V, N))
    b = rng.integers(0, 6, (V, N)) if integer else rng.integers(0, 1000, (V, N))
    m = rng.integers(1, 3, (V, N))
    cum = lambda x: np.concatenate([np.zeros((V, 1), np.uint64), np.cumsum(x, axis=1).astype(np.uint64)], axis=1)
    return dataclasses.replace(prob, PF=cum(f), PB=cum(b), PM=cum(m), blk_flops=f.max(1).astype(np.uint64),
                               blk_bytes=b.max(1).astype(np.uint64), blk_mem=m.max(1).astype(np.uint64))


def bf_value_at(op, v, devs, total, k, mu):
    """min over compositions of blocks 0..total-1 on devs[0..k) of the largest
    stage or link time, with per-layer costs (a stage's cost depends on where
    it starts)."""
    best = INF
    for comp in compositions(total, k):
        worst, j = 0.0, 0
        for t in range(k):
            worst = max(worst, op.stage_cost_at(v, int(devs[t]), j, comp[t], t == mu))
            if t >= 1:
                worst = max(worst, op.link_cost(v, int(devs[t - 1]), int(devs[t])))
            j += comp[t]
        best = min(best, worst)
    return best


def bf_dp_at(op, v, devs, N):
    m = len(devs)
    if m > N:
        return None
    vals = [bf_value_at(op, v, devs, N, m, mu) for mu in range(m)]
    V = min(vals)
    if V == INF:
        return None
    mu = vals.index(V)
    layers = [0] * m
    i = N - 1
    for k in range(m, 1, -1):
        target = bf_value_at(op, v, devs, i + 1, k, mu)
        tau = op.link_cost(v, int(devs[k - 2]), int(devs[k - 1]))
        for j in range(k - 1, i + 1):
            prev = bf_value_at(op, v, devs, j, k - 1, mu)
            c = max(prev, op.stage_cost_at(v, int(devs[k - 1]), j, i - j + 1, mu == k - 1), tau)
            if c == target:
                break
        layers[k - 1] = i - j + 1
        i = j - 1
    layers[0] = i + 1
    return V, mu, layers


@pytest.mark.parametrize("seed", range(24))
def test_layered_dp_matches_brute_force(seed):
    rng = np.random.default_rng(300 + seed)
    N = int(rng.integers(1, 10))
    M = 6
    prob = _layered(tiny_problem(rng, M, N, integer=seed % 4 != 3, head=seed % 5 != 0), rng, integer=seed % 4 != 3)
    op = O.OracleProblem(prob)
    for trial in range(4):
        m = int(rng.integers(1, M + 1))
        devs = rng.permutation(M)[:m]
        v = int(rng.integers(0, prob.V))
        got = op.dp_pipe(v, devs)
        bf = bf_dp_at(op, v, devs, N)
        if bf is None:
            assert not got["ok"]
            continue
        V, mu, layers = bf
        assert got["ok"] and got["V"] == V and got["mu"] == mu and list(got["layers"]) == layers, (devs, v)


def test_layered_with_uniform_sums_is_the_identical_block_model():
    import dataclasses
    for name in ("c1_tiny", "c2"):
        prob = W.make_config(name, P=64)
        V, N = prob.V, prob.N
        ramp = np.arange(N + 1, dtype=np.uint64)[None, :]
        lay = dataclasses.replace(prob, PF=prob.blk_flops[:, None] * ramp, PB=prob.blk_bytes[:, None] * ramp,
                                  PM=prob.blk_mem[:, None] * ramp)
        g = W.random_genomes(prob.M, prob.K_max, 64, seed=4)
        a = O.OracleProblem(prob).eval_population(g, prob.K_max, nthreads=4)
        b = O.OracleProblem(lay).eval_population(g, prob.K_max, nthreads=4)
        for k in ("fitness", "layers", "master", "bsel", "T", "L"):
            assert np.array_equal(a[k], b[k]), (name, k)


def test_layered_prefix_optimum_is_not_monotone():
    """Why blocks of several types need the plain scan: with blocks (light,
    heavy, light) on a fast then a slow device, two blocks cost more than
    three (the slow device must take the heavy block when only two are
    placed).  D(1, 2) = 100 > D(2, 2) = 11; the partition of three blocks
    puts the heavy block on the fast device."""
    # device 0: 1 FLOP/s, device 1: 0.1 FLOP/s; blocks' flops 1, 10, 1
    PF = np.array([[0, 1, 11, 12]], np.uint64)
    zero = np.zeros((1, 4), np.uint64)
    prob = W.make_problem([1.0, 0.1], [1.0, 1.0], [100, 100], np.full((2, 2), np.inf), np.ones((2, 2)), 3,
                          [10], [0], [0], [0], [0], [0], [0], NP=1, ND=1, PF=PF, PB=zero, PM=zero)
    op = O.OracleProblem(prob)
    full = op.dp_pipe(0, [0, 1])
    assert full["ok"] and full["V"] == 11.0 and list(full["layers"]) == [2, 1]
    two = O.OracleProblem(dataclasses_replace(prob, N=2, PF=PF[:, :3], PB=zero[:, :3], PM=zero[:, :3])).dp_pipe(0, [0, 1])
    assert two["V"] == 100.0 and list(two["layers"]) == [1, 1]
    # the per-request latency walks the blocks in order: 11 + 1/0.1
    assert op.latency(0, [0, 1], full["mu"], full["layers"]) == 11.0 + 10.0


def dataclasses_replace(p, **kw):
    import dataclasses
    return dataclasses.replace(p, **kw)
