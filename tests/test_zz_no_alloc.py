"""The allocation-free elite selection against the oracle and the regular path.

e2_select_elites_noalloc exists for callers that cannot allocate device
memory (a CUDA graph being recorded, a host framework whose allocator owns the
device, loops that must not stall on cudaMalloc): it keeps its scratch in a
fixed device array inside the library instead of a caller's workspace.  This
test feeds it populations evaluated on the GPU, with planted duplicate genomes
and a population that is not a multiple of the kernels' block size, and checks
that it picks exactly the elites of the oracle's elite step (the Q best
distinct genomes) for Q = 0, 1, 48 and P, and the elites e2_ga_step picked.
The calls run back to back with different populations, so leftovers of one
call in the shared array cannot leak into the next; the first population is
selected again at the end.
"""
import numpy as np
import pytest

from paper_2606_03770_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _population_with_duplicates(prob, seed):
    g = W.random_genomes(prob.M, prob.K_max, prob.P, seed)
    rng = np.random.default_rng(seed)
    src = rng.integers(0, prob.P, 120)
    dst = rng.integers(0, prob.P, 120)
    for d, s in zip(dst, src):                      # copies, some of them later than the original
        for k in g:
            g[k][d] = g[k][s]
    return g


def test_noalloc_elites_match_the_oracle_and_the_regular_path():
    import torch

    import __graft_entry__ as ge
    ge.build()
    from oracle import oracle as O
    from paper_2606_03770_gb300 import e2ga

    prob = W.make_config("c2", P=1000)
    prob.Q = 48
    eng = e2ga.Engine(prob)
    stream = torch.cuda.current_stream()
    runs = []
    for seed in (5, 6):
        host = _population_with_duplicates(prob, seed)
        eng.eval(genomes=host, parts=False)
        fit = eng.fitness.clone()
        eng.ga_step(17, seed)
        regular, _ = eng.elites()
        torch.cuda.synchronize()
        views = {np.dtype(np.uint16): np.int16, np.dtype(np.uint64): np.int64}
        dev = {k: torch.from_numpy(np.ascontiguousarray(v).view(views.get(v.dtype, v.dtype))).cuda()
               for k, v in host.items()}
        runs.append((host, dev, fit, regular.copy()))
    for host, dev, fit, regular in runs + runs[:1]:
        g = e2ga.e2_genomes(dev["perm"].data_ptr(), dev["sizes"].data_ptr(), dev["nclus"].data_ptr(),
                            dev["roles"].data_ptr())
        fit_h = fit.cpu().numpy()
        for Q in (prob.Q, 0, 1, prob.P):
            out = torch.full((max(Q, 1),), -7, dtype=torch.int32, device="cuda")
            st = e2ga.e2_select_elites_noalloc(g, fit.data_ptr(), prob.P, prob.M, prob.K_max, Q,
                                               out.data_ptr(), stream.cuda_stream)
            assert st == e2ga.E2_OK
            torch.cuda.synchronize()
            got = out.cpu().numpy()
            if Q == 0:
                assert np.all(got == -7)                     # nothing written
                continue
            ga = O._ga_struct(prob.P, prob.M, prob.K_max, Q, prob.tournament, prob.p_cx, prob.p_mut, prob.p_kind)
            assert np.array_equal(got, O.elites(ga, host, fit_h))
            if Q == prob.Q:
                assert np.array_equal(got, regular)
    # sizes beyond the fixed scratch are refused, not run
    host, dev, fit, _ = runs[0]
    g = e2ga.e2_genomes(dev["perm"].data_ptr(), dev["sizes"].data_ptr(), dev["nclus"].data_ptr(),
                        dev["roles"].data_ptr())
    out = torch.zeros(1, dtype=torch.int32, device="cuda")
    st = e2ga.e2_select_elites_noalloc(g, fit.data_ptr(), 65537, prob.M, prob.K_max, 1, out.data_ptr(),
                                       stream.cuda_stream)
    assert st == e2ga.E2_EINVAL
    # host memory is refused as well
    fit_host = fit.cpu()
    st = e2ga.e2_select_elites_noalloc(g, fit_host.data_ptr(), prob.P, prob.M, prob.K_max, 1, out.data_ptr(),
                                       stream.cuda_stream)
    assert st == e2ga.E2_EINVAL
    eng.close()
