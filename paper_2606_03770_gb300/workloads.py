"""Seeded synthetic fleets, links and layer profiles.

This module is the one piece both the CUDA path and the CPU oracle consume.  It
draws inputs only: device capabilities, link bandwidths, congestion factors and
the per-block work of a dense decoder.  None of the planner's arithmetic (stage
cost, link cost, the partition DP, the objective, the genetic operators) lives
here.

The paper profiles per-block latency on real devices with a reduced-block
llama.cpp (Sec. 3.1).  Those profiles are not available, so each device is
described by a compute rate, a memory bandwidth and a memory capacity, and each
block of the model by the FLOPs it executes, the bytes it streams and the bytes
it keeps resident, per inference variant (prefill, or decode with batch b).
Blocks are identical in size and cost, the premise the paper states for fixing
the node order in its DP (Sec. 3.2).

Units: FLOPs, bytes, FLOP/s, bytes/s, tokens.  All integers are Python ints /
numpy uint64 below 2**53 so that both sides convert them to float64 exactly.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

HEAD_DIM = 128


@dataclasses.dataclass
class Problem:
    """One planning instance: fleet, links, layer profile and GA parameters."""

    name: str
    # fleet (M devices)
    rate: np.ndarray  # float64[M] compute rate, FLOP/s
    bw: np.ndarray  # float64[M] memory bandwidth, bytes/s
    mem: np.ndarray  # uint64[M] memory available for the model, bytes
    # links (row = sender, column = receiver)
    link_bw: np.ndarray  # float64[M, M] base link bandwidth, bytes/s
    cong: np.ndarray  # float64[M, M] congestion factor in (0, 1]
    # layer profile: N identical blocks, variant 0 = prefill, v = b >= 1 = decode batch b
    N: int
    blk_flops: np.ndarray  # uint64[V]
    blk_bytes: np.ndarray  # uint64[V]
    blk_mem: np.ndarray  # uint64[V]
    head_flops: np.ndarray  # uint64[V]  LM head + output layer, master only
    head_bytes: np.ndarray  # uint64[V]
    head_mem: np.ndarray  # uint64[V]
    act_bytes: np.ndarray  # uint64[V]  activation bytes of one microbatch crossing a link
    NP: int  # average input tokens per request
    ND: int  # average generated tokens per request
    # objective
    min_tps: float = 7.0
    t_a: float = 1.0
    # roles: 0 = one role bit per replica in the genome; 1 = Alg. 2's brute force
    # over every role assignment of the genome's replicas; 2 = the adapted-SplitWise
    # rule (the strongest replicas prefill)
    role_search: int = 0
    # objective: 0 = the waiting time of Eq. 3-5; 1 = the per-request finishing time
    objective: int = 0
    # genetic algorithm
    P: int = 64
    Q: int = 2
    K_max: int = 2
    G: int = 1
    tournament: int = 4
    p_cx: float = 0.5
    p_mut: float = 0.3
    p_kind: tuple = (0.2, 0.5, 0.15, 0.15)
    redraw: bool = False
    cong_lo: float = 0.2
    cong_hi: float = 1.0
    seed: int = 0
    # GPU-CPU offload: host compute rate (FLOP/s), host memory bandwidth
    # (bytes/s) and host memory for offloaded blocks (bytes) per device; None:
    # no device offloads (0 host memory: a unified-memory device)
    rate_cpu: np.ndarray | None = None
    bw_cpu: np.ndarray | None = None
    mem_cpu: np.ndarray | None = None
    # blocks of several types: per-variant prefix sums [V][N+1] of the blocks'
    # flops, bytes and resident bytes (None: N identical blocks, blk_*)
    PF: np.ndarray | None = None
    PB: np.ndarray | None = None
    PM: np.ndarray | None = None

    @property
    def M(self) -> int:
        return int(self.rate.shape[0])

    @property
    def b_max(self) -> int:
        return int(self.blk_flops.shape[0]) - 1

    @property
    def V(self) -> int:
        return int(self.blk_flops.shape[0])


def _log_uniform(rng, lo, hi, n):
    return np.exp(rng.uniform(math.log(lo), math.log(hi), n))


def _sym(rng, M, draw):
    """Symmetric matrix of per-pair draws; the diagonal is never used by the planner."""
    out = np.ones((M, M), dtype=np.float64)
    iu = np.triu_indices(M, 1)
    vals = draw(len(iu[0]))
    out[iu] = vals
    out[(iu[1], iu[0])] = vals
    return out


def dense_profile(N, d, ffn, kv_heads, vocab, NP, ND, b_max, wbits=16):
    """Per-block work of a dense decoder with ``wbits``-bit weights and fp16 KV cache.

    Block parameters P_l = 2 d^2 + 2 d d_kv + 3 d ffn (q/o, k/v with grouped KV
    heads, gated MLP).  Prefill runs one request of NP tokens; decode variant b
    runs b requests, one token each, against a context of NP + ND tokens.
    """
    d_kv = d if kv_heads is None else kv_heads * HEAD_DIM
    P_l = 2 * d * d + 2 * d * d_kv + 3 * d * ffn
    wbytes = P_l * wbits // 8
    assert wbytes * 8 == P_l * wbits
    ctx = NP + ND
    V = 1 + b_max
    f = np.zeros(V, np.uint64)
    y = np.zeros(V, np.uint64)
    s = np.zeros(V, np.uint64)
    hf = np.zeros(V, np.uint64)
    hy = np.zeros(V, np.uint64)
    hs = np.zeros(V, np.uint64)
    a = np.zeros(V, np.uint64)
    head_params = 2 * d * vocab  # embedding + output projection
    for v in range(V):
        tokens = NP if v == 0 else v
        slots, kv_ctx = (1, NP) if v == 0 else (v, ctx)
        if v == 0:
            f[v] = 2 * P_l * NP + 4 * NP * NP * d
            y[v] = wbytes + NP * 2 * d_kv * 2
        else:
            f[v] = 2 * P_l * v + 4 * v * ctx * d
            y[v] = wbytes + v * ctx * 2 * d_kv * 2
        s[v] = wbytes + slots * kv_ctx * 2 * d_kv * 2
        hf[v] = 2 * d * vocab * tokens
        hy[v] = head_params * wbits // 8
        hs[v] = head_params * wbits // 8
        a[v] = tokens * d * 2
    return dict(blk_flops=f, blk_bytes=y, blk_mem=s, head_flops=hf, head_bytes=hy,
                head_mem=hs, act_bytes=a)


def layered_profile(N, d, ffn, kv_heads, vocab, NP, ND, b_max, wbits=16, window=128, pattern="alternate"):
    """Blocks of two types, as in a model that alternates sliding-window and
    full attention: a sliding-window block attends to (and keeps the KV cache
    of) at most ``window`` positions, a full-attention block to the whole
    context.  Returns the identical-block fields (each the largest block, so
    that range checks stay conservative) plus the per-variant prefix sums
    PF, PB, PM [V][N+1] of the blocks' flops, bytes and resident bytes.
    ``pattern``: "alternate" (sliding on even blocks) or "tail" (the last
    N // 4 blocks full, the rest sliding)."""
    d_kv = d if kv_heads is None else kv_heads * HEAD_DIM
    P_l = 2 * d * d + 2 * d * d_kv + 3 * d * ffn
    wbytes = P_l * wbits // 8
    assert wbytes * 8 == P_l * wbits
    ctx = NP + ND
    V = 1 + b_max
    base = dense_profile(N, d, ffn, kv_heads, vocab, NP, ND, b_max, wbits)
    PF = np.zeros((V, N + 1), np.uint64)
    PB = np.zeros((V, N + 1), np.uint64)
    PM = np.zeros((V, N + 1), np.uint64)
    for v in range(V):
        f, y, s_ = [], [], []
        for l in range(N):
            sliding = (l % 2 == 0) if pattern == "alternate" else (l < N - N // 4)
            if v == 0:
                seen = min(NP, window) if sliding else NP
                f.append(2 * P_l * NP + 4 * NP * seen * d)
                kv = min(NP, window) if sliding else NP
                y.append(wbytes + kv * 2 * d_kv * 2)
                s_.append(wbytes + kv * 2 * d_kv * 2)
            else:
                seen = min(ctx, window) if sliding else ctx
                f.append(2 * P_l * v + 4 * v * seen * d)
                y.append(wbytes + v * seen * 2 * d_kv * 2)
                s_.append(wbytes + v * seen * 2 * d_kv * 2)
        PF[v, 1:] = np.cumsum(np.array(f, dtype=np.uint64))
        PB[v, 1:] = np.cumsum(np.array(y, dtype=np.uint64))
        PM[v, 1:] = np.cumsum(np.array(s_, dtype=np.uint64))
        base["blk_flops"][v] = max(f)
        base["blk_bytes"][v] = max(y)
        base["blk_mem"][v] = max(s_)
    base.update(PF=PF, PB=PB, PM=PM)
    return base


# Fleet and model shapes of the five workloads the planner is measured on.  The
# 32-block model keeps fp16 weights; the 80- and 126-block models carry 4-bit
# weights, the precision of the models the paper deploys (Q4_K_M, MXFP4), without
# which no decode replica of these fleets reaches the 7 tokens/s floor.
CONFIGS = {
    "c1_tiny": dict(M=8, tflops=("log", 2, 30), mem_gb=(4, 16), link=("uniform", 0.1, 10),
                    cong=(0.3, 1.0), model=dict(N=32, d=4096, ffn=11008, kv_heads=None, vocab=32000, wbits=16),
                    prompt=("fixed", 512), K_max=2, P=64, G=1),
    "c2": dict(M=32, tflops=("log", 2, 30), mem_gb=(4, 32), link=("uniform", 0.1, 10),
               cong=(0.3, 1.0), model=dict(N=80, d=8192, ffn=28672, kv_heads=8, vocab=128256, wbits=4),
               prompt=("mean", 256, 2048), K_max=8, P=1024, G=10),
    "c3": dict(M=128, tflops=("log", 2, 30), mem_gb=(4, 32), link=("uniform", 0.1, 10),
               cong=(0.3, 1.0), model=dict(N=80, d=8192, ffn=28672, kv_heads=8, vocab=128256, wbits=4),
               prompt=("mean", 256, 2048), K_max=16, P=4096, G=50, redraw=(0.2, 1.0)),
    "c4": dict(M=512, tflops=("log", 1, 60), mem_gb=(2, 64), link=("log", 0.05, 25),
               cong=(0.3, 1.0), model=dict(N=126, d=16384, ffn=53248, kv_heads=8, vocab=128256, wbits=4),
               prompt=("mean", 256, 4096), K_max=64, P=16384, G=1),
    "c5": dict(M=256, tflops=("log", 2, 30), mem_gb=(4, 32), link=("uniform", 0.1, 10),
               cong=(0.3, 1.0), model=dict(N=80, d=8192, ffn=28672, kv_heads=8, vocab=128256, wbits=4),
               prompt=("mean", 256, 2048), K_max=32, P=8192, G=200, p_mut=0.01),
}

DEVICE_BW_GBS = (50.0, 800.0)  # device memory bandwidth, log-uniform (not given by the configs)
B_MAX = 8
# Host side of GPU-CPU offload (the paper's fleet mixes discrete GPUs with host
# RAM and unified-memory devices): half the devices are unified (no host memory
# for blocks); the others offload to U[16, 128] GB of host RAM, run offloaded
# blocks at log-U[0.2, 2] TFLOP/s and stream them at log-U[20, 120] GB/s.
HOST_MEM_GB = (16.0, 128.0)
HOST_TFLOPS = (0.2, 2.0)
HOST_BW_GBS = (20.0, 120.0)


def offload_fleet(M: int, seed: int):
    """Host rates, bandwidths and memories of an offloading fleet of M devices,
    from a generator of its own (the fleet's other draws do not move)."""
    rng = np.random.Generator(np.random.Philox(key=seed + 104729))
    unified = rng.uniform(0.0, 1.0, M) < 0.5
    mem = np.array([0 if u else int(round(x * 1e9)) for u, x in zip(unified, rng.uniform(*HOST_MEM_GB, M))],
                   dtype=np.uint64)
    rate = _log_uniform(rng, HOST_TFLOPS[0], HOST_TFLOPS[1], M) * 1e12
    bw = _log_uniform(rng, HOST_BW_GBS[0], HOST_BW_GBS[1], M) * 1e9
    return rate, bw, mem


def make_config(name: str, seed: int = 0, P: int | None = None, offload: bool = False,
                layered: str | None = None) -> Problem:
    """Draw the named workload with a numpy Philox generator keyed by ``seed``
    (with ``offload``, plus the host side of GPU-CPU offload per device; with
    ``layered`` = "alternate" or "tail", the model's blocks are of two types,
    sliding-window and full attention, given as per-layer prefix sums)."""
    c = CONFIGS[name]
    rng = np.random.Generator(np.random.Philox(key=seed))
    M = c["M"]
    kind, lo, hi = c["tflops"]
    tflops = _log_uniform(rng, lo, hi, M) if kind == "log" else rng.uniform(lo, hi, M)
    rate = tflops * 1e12
    bw = _log_uniform(rng, DEVICE_BW_GBS[0], DEVICE_BW_GBS[1], M) * 1e9
    mem = np.array([int(round(x * 1e9)) for x in rng.uniform(c["mem_gb"][0], c["mem_gb"][1], M)],
                   dtype=np.uint64)
    lk, llo, lhi = c["link"]
    if lk == "log":
        gbps = _sym(rng, M, lambda n: _log_uniform(rng, llo, lhi, n))
    else:
        gbps = _sym(rng, M, lambda n: rng.uniform(llo, lhi, n))
    link_bw = gbps * 1.25e8
    np.fill_diagonal(link_bw, np.inf)
    cong = _sym(rng, M, lambda n: rng.uniform(c["cong"][0], c["cong"][1], n))
    pk = c["prompt"]
    if pk[0] == "fixed":
        NP = int(pk[1])
    else:
        NP = int(round(float(np.mean(rng.integers(pk[1], pk[2] + 1, 1000)))))
    ND = NP  # generated tokens: input/generated ratios of 0.77-1.65 are reported, take 1
    if layered:
        prof = layered_profile(NP=NP, ND=ND, b_max=B_MAX, pattern=layered, **c["model"])
    else:
        prof = dense_profile(NP=NP, ND=ND, b_max=B_MAX, **c["model"])
    P_ = int(P if P is not None else c["P"])
    redraw = c.get("redraw")
    host = dict(zip(("rate_cpu", "bw_cpu", "mem_cpu"), offload_fleet(M, seed))) if offload else {}
    return Problem(
        name=name, rate=rate, bw=bw, mem=mem, link_bw=link_bw, cong=cong,
        N=c["model"]["N"], NP=NP, ND=ND, P=P_, Q=int(math.ceil(P_ / 32)), K_max=c["K_max"],
        G=c["G"], p_mut=c.get("p_mut", 0.3), redraw=redraw is not None,
        cong_lo=(redraw or (0.2, 1.0))[0], cong_hi=(redraw or (0.2, 1.0))[1], seed=seed,
        **prof, **host)


def make_problem(rate, bw, mem, link_bw, cong, N, blk_flops, blk_bytes, blk_mem, head_flops,
                 head_bytes, head_mem, act_bytes, NP, ND, name="custom", **kw) -> Problem:
    """Build a Problem from explicit arrays (hand-made cases, edge cases)."""
    f64 = lambda x: np.ascontiguousarray(np.asarray(x, dtype=np.float64))
    u64 = lambda x: np.ascontiguousarray(np.asarray(x, dtype=np.uint64))
    for k, conv in (("rate_cpu", f64), ("bw_cpu", f64), ("mem_cpu", u64), ("PF", u64), ("PB", u64), ("PM", u64)):
        if kw.get(k) is not None:
            kw[k] = conv(kw[k])
    return Problem(name=name, rate=f64(rate), bw=f64(bw), mem=u64(mem), link_bw=f64(link_bw),
                   cong=f64(cong), N=int(N), blk_flops=u64(blk_flops), blk_bytes=u64(blk_bytes),
                   blk_mem=u64(blk_mem), head_flops=u64(head_flops), head_bytes=u64(head_bytes),
                   head_mem=u64(head_mem), act_bytes=u64(act_bytes), NP=int(NP), ND=int(ND), **kw)


def random_genomes(M: int, K_max: int, P: int, seed: int, max_clusters: int | None = None):
    """Valid random genomes (uniform permutation, random composition, random roles).

    Used to feed both sides the same population for evaluation-only parity; the
    GA's own initialisation is part of the method and is not drawn here.
    """
    rng = np.random.Generator(np.random.Philox(key=seed + 7919))
    kmax = min(K_max, M) if max_clusters is None else min(max_clusters, K_max, M)
    perm = np.zeros((P, M), np.uint16)
    sizes = np.zeros((P, K_max), np.uint16)
    nclus = np.zeros(P, np.uint8)
    roles = np.zeros(P, np.uint64)
    for g in range(P):
        perm[g] = rng.permutation(M)
        R = int(rng.integers(1, kmax + 1))
        cuts = np.sort(rng.choice(np.arange(1, M), R - 1, replace=False)) if R > 1 else np.array([], int)
        edges = np.concatenate([[0], cuts, [M]])
        sizes[g, :R] = np.diff(edges)
        nclus[g] = R
        bits = int(rng.integers(0, 1 << min(R, 62)))
        if R > 62:
            bits |= int(rng.integers(0, 1 << (R - 62))) << 62
        roles[g] = np.uint64(bits)
    return dict(perm=perm, sizes=sizes, nclus=nclus, roles=roles)
