"""NaN inputs on the GPU paths: the predictors' ReLU keeps NaN, so a NaN weight of
model 0 makes every candidate's objective NaN, and a candidate whose objective is NaN
is infeasible (scored -inf, never counted, never in a top-k).  The oracle's pin of
the same reading is test_oracle_pins.test_nan_weights_make_candidates_infeasible."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

pytestmark = pytest.mark.gpu

EMPTY = 2 ** 64 - 1


@pytest.fixture(scope="module")
def mf():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_02109_gb300 import build
    build.build()
    from paper_2609_02109_gb300 import mf as mod
    return mod


def _with_nan(prob, pos):
    """A NaN in W1[0][0] or in b3[1] (the latency bias) of model 0."""
    p = dict(prob)
    p["weights"] = p["weights"].copy()
    per = W.param_count(int(p["d_local"]), int(p["hidden1"]), int(p["hidden2"]))
    p["weights"][0 if pos == "W1" else per - 1] = np.nan
    return p


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
@pytest.mark.parametrize("pos", ["W1", "b3"])
def test_nan_weight_makes_every_candidate_infeasible(mf, oracle_mod, precision, pos):
    import torch
    prob = _with_nan(W.tiny(), pos)
    assert oracle_mod.Oracle(prob).exhaustive(4)[2] == 0
    with mf.Context(prob, precision=precision) as ctx:
        res = ctx.search(4)
        assert res["count"] == 0
        assert res["best_idx"] == EMPTY and res["best_score"] == -np.inf
        assert np.all(res["topk_idx"] == np.uint64(EMPTY)) and np.all(res["topk_score"] == -np.inf)
        idx = torch.arange(ctx.space_size, dtype=torch.int64, device="cuda")
        score, feas = ctx.score_batch(idx)
        torch.cuda.synchronize()
        assert torch.all(score == -float("inf")) and not feas.any()


@pytest.mark.parametrize("pos", ["W1", "b3"])
def test_nan_weight_gives_minus_infinity_fitness_and_the_oracle_s_ga_run(mf, oracle_mod, pos):
    """mf_ga_generation scores every individual -inf; a whole decision (the cooperative
    kernel: N = 5, 12->64->64->2) then runs on an all -inf landscape, where every
    tournament and the elite fall to the lowest slot drawn, and must return the
    oracle's genome."""
    import torch
    prob = _with_nan(W.paper_scale(), pos)
    o = oracle_mod.Oracle(prob)
    g = dict(W.GA_PARAMS, gens=12)
    with mf.Context(prob) as ctx:
        pop = torch.from_numpy(o.ga_init(g, 5)).cuda()
        fit = ctx.ga_generation(pop)
        torch.cuda.synchronize()
        assert torch.all(fit == -float("inf"))
        for seed in (3, 1000):
            J, genome = ctx.ga_run(g, seed)
            Jo, go = o.ga_run(g, seed)
            assert J == -np.inf and Jo == -np.inf
            assert list(genome) == list(go)
