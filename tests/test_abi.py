"""The C ABI without a GPU: the library builds, loads and exports every symbol
include/e2ga.h declares, and e2_create rejects invalid inputs with a status
before it touches the device."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2606_03770_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2606_03770_gb300 import build, e2ga
    build.build()
    return e2ga.load()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "e2ga.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(e2_[a-z_]+)\s*\(", src)))


def test_exports_every_declared_symbol(lib):
    from paper_2606_03770_gb300 import e2ga
    names = declared_functions()
    assert len(names) >= 14
    for n in names:
        assert hasattr(lib, n), n
        assert n in e2ga.SIGNATURES, n
    assert set(e2ga.SIGNATURES) == set(names)


def declared_struct_fields(name):
    src = open(os.path.join(ROOT, "include", "e2ga.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    body = re.search(r"typedef struct \{([^}]*)\}\s*" + name + r"\s*;", src).group(1)
    return [(t, n) for t, n in re.findall(r"(\w+)\s*\*?\s*(\w+)\s*;", body)]


@pytest.mark.parametrize("name", ["e2_devices", "e2_layer_profile", "e2_params", "e2_stats", "e2_genomes",
                                  "e2_partitions"])
def test_binding_structs_follow_the_header(name):
    """The ctypes mirrors of the header's structs: same fields in the same
    order, with the same widths."""
    from paper_2606_03770_gb300 import e2ga
    widths = {"int32_t": 4, "uint32_t": 4, "int": 4, "uint64_t": 8, "int64_t": 8, "double": 8, "float": 4}
    decl = declared_struct_fields(name)
    mine = getattr(e2ga, name)._fields_
    assert len(decl) == len(mine), (decl, mine)
    src = open(os.path.join(ROOT, "include", "e2ga.h")).read()
    for (t, n), (pn, pt) in zip(decl, mine):
        assert pn.rstrip("_") == n, (n, pn)
        pointer = re.search(r"\b" + t + r"\s*\*\s*" + n + r"\s*;", src) is not None
        if pointer:
            assert pt is C.c_void_p or issubclass(pt, C._Pointer), (n, pt)
        else:
            assert C.sizeof(pt) == widths[t], (n, t, pt)


def test_workspace_bytes(lib):
    from paper_2606_03770_gb300 import e2ga
    for name in ("c1_tiny", "c2", "c4"):
        p = W.make_config(name)
        n = e2ga.e2_workspace_bytes(p.M, p.N, p.b_max, p.P, p.Q, p.K_max)
        assert n > 0 and n % 256 == 0
        # the population and per-replica results dominate; tables scale with V*M*(M+N)
        assert n >= p.P * (2 * p.M + 32)
    assert e2ga.e2_workspace_bytes(0, 10, 8, 10, 1, 2) == 0
    assert e2ga.e2_workspace_bytes(8, 10, 8, 10, 11, 2) == 0      # Q > P
    assert e2ga.e2_workspace_bytes(8, 10, 8, 10, 1, 65) == 0      # K_max > 64
    # work items P * K_max * (b_max + 1) must stay below 2^31
    assert e2ga.e2_workspace_bytes(8, 10, 63, (1 << 22) - 1, 1, 8) > 0
    assert e2ga.e2_workspace_bytes(8, 10, 63, (1 << 22), 1, 8) == 0


def _structs(prob):
    from paper_2606_03770_gb300 import e2ga
    keep = []

    def p(a):
        keep.append(a)
        return a.ctypes.data

    f64 = lambda x: np.ascontiguousarray(x, dtype=np.float64)
    u64 = lambda x: np.ascontiguousarray(x, dtype=np.uint64)
    d = e2ga.e2_devices(prob.M, p(f64(prob.rate)), p(f64(prob.bw)), p(u64(prob.mem)))
    l = e2ga.e2_links(p(f64(prob.link_bw)), p(f64(prob.cong)), prob.cong_lo, prob.cong_hi)
    pf = e2ga.e2_layer_profile(prob.N, prob.b_max, *[p(u64(getattr(prob, k))) for k in (
        "blk_flops", "blk_bytes", "blk_mem", "head_flops", "head_bytes", "head_mem", "act_bytes")], prob.NP, prob.ND)
    pr = e2ga.e2_params(prob.P, prob.Q, prob.K_max, prob.tournament, prob.min_tps, prob.t_a, prob.p_cx,
                        prob.p_mut, *prob.p_kind[:3], prob.role_search, prob.objective)
    return d, l, pf, pr, keep


BAD = {
    "role search mode": lambda p: setattr(p, "role_search", 3),
    "objective": lambda p: setattr(p, "objective", 2),
    "role search with a large batch": lambda p: (setattr(p, "role_search", 1), setattr(p, "blk_flops", np.ones(70, np.uint64))),
    "negative rate": lambda p: p.rate.__setitem__(0, -1.0),
    "nan bandwidth": lambda p: p.bw.__setitem__(1, np.nan),
    "zero link": lambda p: p.link_bw.__setitem__((0, 1), 0.0),
    "inf congestion": lambda p: p.cong.__setitem__((2, 1), np.inf),
    "Q > P": lambda p: setattr(p, "Q", p.P + 1),
    "K_max 0": lambda p: setattr(p, "K_max", 0),
    "probability > 1": lambda p: setattr(p, "p_cx", 1.5),
    "negative T_a": lambda p: setattr(p, "t_a", -1.0),
    "tournament 0": lambda p: setattr(p, "tournament", 0),
    "2^53 overflow": lambda p: p.blk_flops.__setitem__(0, np.uint64(2 ** 52)),
}


@pytest.mark.parametrize("what", sorted(BAD))
def test_create_rejects_invalid_inputs_without_a_device(lib, what):
    from paper_2606_03770_gb300 import e2ga
    prob = W.make_config("c1_tiny")
    BAD[what](prob)
    d, l, pf, pr, keep = _structs(prob)
    ws = (C.c_uint8 * 1024)()
    ctx = C.c_void_p()
    st = lib.e2_create(C.byref(d), C.byref(l), C.byref(pf), C.byref(pr), C.addressof(ws), 1024, None, C.byref(ctx))
    assert st == e2ga.E2_EINVAL
    assert ctx.value is None
    assert e2ga.e2_last_error(None) != ""


def test_create_rejects_short_workspace(lib):
    from paper_2606_03770_gb300 import e2ga
    prob = W.make_config("c1_tiny")
    d, l, pf, pr, keep = _structs(prob)
    buf = (C.c_uint8 * 4096)()
    base = (C.addressof(buf) + 255) & ~255
    ctx = C.c_void_p()
    st = lib.e2_create(C.byref(d), C.byref(l), C.byref(pf), C.byref(pr), base, 1024, None, C.byref(ctx))
    assert st == e2ga.E2_ENOMEM
    st = lib.e2_create(C.byref(d), C.byref(l), C.byref(pf), C.byref(pr), base + 8, 10 ** 9, None, C.byref(ctx))
    assert st == e2ga.E2_EINVAL                          # misaligned workspace


def test_null_context_calls_are_rejected(lib):
    from paper_2606_03770_gb300 import e2ga
    assert lib.e2_init_population(None, 1) == e2ga.E2_EINVAL
    assert lib.e2_ga_step(None, 1, 1) == e2ga.E2_EINVAL
    assert lib.e2_eval_population(None, None, None, None) == e2ga.E2_EINVAL
    assert lib.e2_destroy(None) == e2ga.E2_OK
    assert lib.e2_set_timing_events(None, None, None) == e2ga.E2_EINVAL
    assert lib.e2_run_generation(None, 1, 1) == e2ga.E2_EINVAL
    assert lib.e2_get_results(None, None, None) == e2ga.E2_EINVAL
    assert lib.e2_run_generation_io(None, None, 1, 1, None, None) == e2ga.E2_EINVAL
    assert e2ga.e2_strerror(e2ga.E2_ESTATE) == "call out of order"


def test_binding_fails_loudly_without_library(tmp_path):
    from paper_2606_03770_gb300 import e2ga
    saved = e2ga._lib
    e2ga._lib = None
    try:
        with pytest.raises(RuntimeError, match="not built"):
            e2ga.load(str(tmp_path / "missing.so"))
    finally:
        e2ga._lib = saved
