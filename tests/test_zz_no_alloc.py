"""The allocation-free elite selection against the regular one.

e2_select_elites_noalloc exists for callers that cannot allocate device
memory (a CUDA graph being recorded, a host framework whose allocator owns the
device, loops that must not stall on cudaMalloc): it keeps its scratch in a
fixed device array inside the library instead of a caller's workspace.  This
test feeds it populations evaluated by the regular path and checks that it
picks exactly the elites e2_ga_step picked, on two calls in a row with
different populations (so leftovers of the first call in the shared array
cannot leak into the second), and once more on the first population.
"""
import numpy as np
import pytest

from paper_2606_03770_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _regular_elites(eng, seed, gen):
    """Population and fitness on the device before the step, and the elites the
    regular path chose for them."""
    import torch
    P, M, K = eng.P, eng.M, eng.K
    pop = dict(perm=torch.empty((P, M), dtype=torch.int16, device="cuda"),
               sizes=torch.empty((P, K), dtype=torch.int16, device="cuda"),
               nclus=torch.empty(P, dtype=torch.uint8, device="cuda"),
               roles=torch.empty(P, dtype=torch.int64, device="cuda"))
    eng.eval(parts=False)
    eng.get_population(pop)
    fit = eng.fitness.clone()
    eng.ga_step(seed, gen)
    idx, _ = eng.elites()
    torch.cuda.synchronize()
    return pop, fit, idx


def test_noalloc_elites_match_the_regular_path():
    import torch

    import __graft_entry__ as ge
    ge.build()
    from paper_2606_03770_gb300 import e2ga

    prob = W.make_config("c2", P=1024)
    prob.Q = 48
    eng = e2ga.Engine(prob)
    eng.init_population(17)
    runs = [_regular_elites(eng, 17, 1), _regular_elites(eng, 17, 2)]
    stream = torch.cuda.current_stream()
    for pop, fit, want in runs + runs[:1]:
        out = torch.full((prob.Q,), -1, dtype=torch.int32, device="cuda")
        g = e2ga.e2_genomes(pop["perm"].data_ptr(), pop["sizes"].data_ptr(), pop["nclus"].data_ptr(),
                            pop["roles"].data_ptr())
        st = e2ga.e2_select_elites_noalloc(g, fit.data_ptr(), prob.P, prob.M, prob.K_max, prob.Q,
                                           out.data_ptr(), stream.cuda_stream)
        assert st == e2ga.E2_OK
        torch.cuda.synchronize()
        assert np.array_equal(out.cpu().numpy(), want)
    # sizes beyond the fixed scratch are refused, not run
    pop, fit, _ = runs[0]
    g = e2ga.e2_genomes(pop["perm"].data_ptr(), pop["sizes"].data_ptr(), pop["nclus"].data_ptr(),
                        pop["roles"].data_ptr())
    st = e2ga.e2_select_elites_noalloc(g, fit.data_ptr(), 65537, prob.M, prob.K_max, 1, out.data_ptr(),
                                       stream.cuda_stream)
    assert st == e2ga.E2_EINVAL
    eng.close()
