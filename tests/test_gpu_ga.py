"""A whole GA decision on the GPU (mf_ga_run) against the oracle's GA, bit for bit.

On a general landscape a GA trajectory is not reproducible across implementations:
fp32 and fp64 fitness differ in the last bits, and one flipped tournament changes
every later generation.  The integer landscapes used here have every predictor
output, objective value and constraint sum an exact small integer, so any correct
evaluation order gives the same fitness and the device run must reproduce the
oracle's run exactly: the same best genome and the same fitness.  That pins the
initial population, every draw of the tournaments, crossover and mutation, the
elitism and tie rules, the double-buffered populations and (for the cooperative
kernel) the grid barrier between generations.

The cases cover both implementations of mf_ga_run: the single cooperative kernel
(one CTA per slice of at most 8 individuals, fp32 12->64->64->2 predictors) and
the CUDA-graph fallback (here: a population above 8 per SM)."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

pytestmark = pytest.mark.gpu

MAX_SLICE = 8  # individuals per CTA of the cooperative kernel


@pytest.fixture(scope="module")
def mf():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_02109_gb300 import build
    build.build()
    from paper_2609_02109_gb300 import mf as mod
    return mod


def _sms():
    import torch
    return torch.cuda.get_device_properties(0).multi_processor_count


CASES = {
    # name: (options, landscape seed, VRAM cap, objective, GA parameters)
    "paper_shape_pop1024": ([12, 9, 9, 9, 9], 5, 30.0, "weighted_thr", dict(W.GA_PARAMS)),
    "no_elitism": ([12, 9, 9, 9, 9], 5, 30.0, "weighted_thr", dict(W.GA_PARAMS, elitism=0, gens=40)),
    "slice_of_one": ([16] * 4, 6, 25.0, "weighted_thr", dict(W.GA_PARAMS, pop=100, gens=60)),
    "eight_models_full_slices": ([5] * 8, 7, 45.0, "soft_lat",
                                 dict(W.GA_PARAMS, pop=8 * 152, gens=20, tournament=3)),
    "one_model": ([200], 8, 9.0, "weighted_thr", dict(W.GA_PARAMS, pop=50, gens=25, mutation_p=0.2)),
    "pop_two_one_gen": ([6, 7, 8], 9, 20.0, "weighted_thr", dict(W.GA_PARAMS, pop=2, gens=1)),
    "single_generation": ([12, 9, 9, 9, 9], 5, 30.0, "weighted_thr", dict(W.GA_PARAMS, gens=1)),
    # the predictors see the candidate's own aggregate (W1's aggregate columns in use,
    # unscaled): the cooperative kernel's coupled fitness, not only its winner
    "coupled_paper_shape": ([12, 9, 9, 9, 9], 5, 30.0, "weighted_thr", dict(W.GA_PARAMS), True),
    "coupled_four_models": ([16] * 4, 6, 25.0, "soft_lat", dict(W.GA_PARAMS, pop=100, gens=60), True),
    # eight models take a whole SM per CTA: a population above 8 per SM cannot be resident
    "graph_fallback_pop_over_8_per_sm": ([5] * 8, 7, 45.0, "weighted_thr",
                                         dict(W.GA_PARAMS, pop=9 * 160, gens=12)),
}


def _problem(name):
    opts, seed, cap, objective = CASES[name][:4]
    coupled = len(CASES[name]) > 5 and CASES[name][5]
    return W.integer_landscape(opts, seed, cap, objective=objective,
                               soft_penalty=0.5 if objective == "soft_lat" else 0.0, coupled=coupled)


@pytest.mark.parametrize("name", list(CASES))
def test_ga_run_reproduces_oracle_run_exactly(mf, oracle_mod, name):
    prob = _problem(name)
    g = CASES[name][4]
    o = oracle_mod.Oracle(prob)
    persistent = not name.startswith("graph_fallback")
    assert persistent or -(-g["pop"] // _sms()) > MAX_SLICE
    with mf.Context(prob) as ctx:
        for seed in (1000, 1001, 2 ** 40 + 3):
            J, genome = ctx.ga_run(g, seed)
            Jo, go = o.ga_run(g, seed)
            assert list(genome) == list(go), (seed, genome, go)
            assert J == Jo, (seed, J, Jo)
            assert ctx.stats()["kernel_launches_last"] == (1 if persistent else 3 * g["gens"] + 1)


def test_repeated_runs_and_seeds(mf, oracle_mod):
    """The seed is read from device memory at each launch: alternating seeds on one
    context give the oracle's answer for each, and a repeated seed repeats it."""
    prob = _problem("paper_shape_pop1024")
    g = dict(W.GA_PARAMS, gens=30)
    o = oracle_mod.Oracle(prob)
    with mf.Context(prob) as ctx:
        runs = [(sd, ctx.ga_run(g, sd)) for sd in (7, 8, 7, 9)]
    for sd, (J, genome) in runs:
        Jo, go = o.ga_run(g, sd)
        assert J == Jo and list(genome) == list(go), sd
