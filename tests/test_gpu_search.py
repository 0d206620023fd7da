"""End-to-end schedule search on the GPU: fitness = -dev_l2 of evo_denoise_population
(quick: 2 observations; formal: 4 others), guided initial individuals from the
GPU redundancy map of the all-refresh trace.  The library's search and the
oracle search, driven by the same (deterministic) GPU fitness, must agree
exactly; the result keeps the budget and is no worse than the best initial
individual."""
import numpy as np
import pytest

from oracle.evo_search import Search
from paper_2607_20293_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as _t
    if not _t.cuda.is_available():
        pytest.skip("no CUDA device")
    return _t


@pytest.fixture(scope="module")
def B(torch):
    from paper_2607_20293_gb300 import binding, build
    build.build()
    binding.load()
    return binding


def test_search_with_population_fitness(torch, B):
    cfg = synth.config("tiny")
    W = synth.make_weights(cfg, 0)
    U, T, H, E = 3 * cfg["n_layer"], cfg["n_steps"], cfg["horizon"], cfg["n_emb"]
    P_max = 12
    ev = B.Evo(cfg, W, (P_max + 1) * 4)
    sets = {}
    for name, n, seed in (("quick", 2, 30), ("formal", 4, 40)):
        sets[name] = (torch.from_numpy(synth.make_obs(cfg, n, seed)).cuda(),
                      torch.from_numpy(synth.make_noise(cfg, n, seed + 1)).cuda())

    def fitness(which):
        obs, noise = sets[which]

        def f(S):
            _, dev = ev.population(obs, noise, S.astype(np.uint8), want_actions=False)
            return [-float(v) for v in dev.cpu().numpy()]
        return f

    # redundancy map from the all-refresh trace of the formal observations
    obs, noise = sets["formal"]
    tr = torch.zeros((T, U, 4, H, E), device="cuda")
    ev.denoise(obs, noise, np.ones((U, T), np.uint8), trace=tr)
    d = B.redundancy_map(tr, "cosine").cpu().numpy()

    kw = dict(population=P_max, elites=4, generations=5, guided=6, early_stop=True, q_base=-0.02, delta_acc=0.01,
              seed=11)
    K = 24
    got = B.search(U, T, K, fitness("quick"), formal=fitness("formal"), d_map=d, **kw)
    want = Search(U, T, K, **kw).run(fitness("quick"), formal=fitness("formal"), d_map=d)
    assert np.array_equal(got[0], want[0]) and got[1] == want[1] and got[2] == want[2]
    assert got[0].sum() == K
    first = Search(U, T, K, **dict(kw, generations=1, early_stop=False)).run(fitness("quick"), d_map=d)
    if not got[2]["stopped_early"]:
        assert got[1] >= first[1]
