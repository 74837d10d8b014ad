"""Pins of the oracle's GA operators (Sec. IV-C: tournament selection,
crossover, mutation, elitism) by properties that any correct implementation of
the stated operators must have.  The whole-GA trajectory is not pinned beyond
these operator properties (a fitness difference of one ulp can flip a
tournament)."""
import math

import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W


def _ga(**kw):
    g = dict(W.GA_PARAMS)
    g.update(kw)
    return g


@pytest.fixture(scope="module")
def prob():
    return W.paper_scale()


def test_rng_counter_fields_are_distinct(oracle_mod):
    seen = set()
    for gen in (0, 1, 99):
        for slot in (0, 1, 1023, 2 ** 20 - 1):
            for purpose in range(6):
                for j in (0, 1, 255):
                    seen.add(oracle_mod.rng(5, gen, slot, purpose, j))
    assert len(seen) == 3 * 4 * 6 * 3


def test_init_is_uniform_over_each_option_range(oracle_mod, prob):
    o = oracle_mod.Oracle(prob)
    pop = o.ga_init(_ga(pop=20000), seed=3)
    ks = prob["n_options"]
    assert pop.shape == (20000, 5)
    for i, k in enumerate(ks):
        assert pop[:, i].min() == 0 and pop[:, i].max() == k - 1
        counts = np.bincount(pop[:, i], minlength=k)
        exp = 20000 / k
        chi2 = float(((counts - exp) ** 2 / exp).sum())
        assert chi2 < k + 8 * math.sqrt(2 * k)  # loose chi-square bound


def test_elitism_keeps_the_fittest_lowest_slot(oracle_mod, prob):
    o = oracle_mod.Oracle(prob)
    g = _ga(pop=64)
    pop = o.ga_init(g, seed=1)
    fit = np.linspace(-1, 1, 64)
    fit[[17, 40]] = 5.0  # tie: slot 17 must win
    nxt = o.ga_step(g, 1, 0, pop, fit)
    assert list(nxt[0]) == list(pop[17])
    g0 = _ga(pop=64, elitism=0)
    nxt0 = o.ga_step(g0, 1, 0, pop, fit)
    assert np.array_equal(nxt0[1:], nxt[1:])  # children do not depend on elitism


def test_children_come_from_two_parents_without_mutation(oracle_mod):
    """With p_m = 0 every child gene is copied from one of two parents.  Slot s
    carries genome (s, s, ..., s), so each child names at most two slots."""
    p = W.make_problem([256] * 6, 8, 16, 0, 5, 1e9)
    o = oracle_mod.Oracle(p)
    g = _ga(pop=256, mutation_p=0.0)
    pop = np.repeat(np.arange(256, dtype=np.int32)[:, None], 6, axis=1)
    fit = np.arange(256, dtype=np.float64)
    nxt = o.ga_step(g, 9, 3, pop, fit)
    mixed = 0
    for c in range(1, 256):
        src = set(nxt[c].tolist())
        assert len(src) <= 2
        mixed += len(src) == 2
    # uniform crossover of two distinct parents gives a mix with prob 1 - 2 / 2**6
    assert mixed > 0.8 * 255
    # tournament of 4 over fitness = slot: the winner is the max of 4 uniform
    # draws, mean about 4/5 of the range
    parents = np.array([v for c in range(1, 256) for v in set(nxt[c].tolist())])
    assert 0.74 * 255 < parents.mean() < 0.86 * 255


def test_tournament_of_one_is_uniform(oracle_mod):
    p = W.make_problem([256], 8, 16, 0, 5, 1e9)
    o = oracle_mod.Oracle(p)
    g = _ga(pop=256, tournament=1, mutation_p=0.0)
    pop = np.arange(256, dtype=np.int32)[:, None]
    nxt = o.ga_step(g, 2, 0, pop, np.arange(256, dtype=np.float64))
    assert 0.4 * 255 < nxt[1:, 0].mean() < 0.6 * 255


def test_mutation_rate(oracle_mod, prob):
    """Identical parents: a gene differs from the parent exactly when it mutated to
    another value, with probability p_m * (1 - 1/K_i)."""
    o = oracle_mod.Oracle(prob)
    P = 8192
    g = _ga(pop=P, mutation_p=0.05)
    pop = np.tile(np.array([3, 4, 5, 6, 7], dtype=np.int32), (P, 1))
    nxt = o.ga_step(g, 11, 7, pop, np.zeros(P))
    ks = prob["n_options"]
    for i, k in enumerate(ks):
        rate = float((nxt[1:, i] != pop[0, i]).mean())
        exp = 0.05 * (1 - 1 / k)
        sd = math.sqrt(exp * (1 - exp) / (P - 1))
        assert abs(rate - exp) < 5 * sd
        assert nxt[:, i].min() >= 0 and nxt[:, i].max() < k


def test_full_mutation_is_uniform(oracle_mod, prob):
    o = oracle_mod.Oracle(prob)
    P = 12000
    g = _ga(pop=P, mutation_p=1.0, elitism=0)
    pop = np.zeros((P, 5), dtype=np.int32)
    nxt = o.ga_step(g, 4, 0, pop, np.zeros(P))
    k = int(prob["n_options"][0])
    counts = np.bincount(nxt[:, 0], minlength=k)
    exp = P / k
    assert float(((counts - exp) ** 2 / exp).sum()) < k + 8 * math.sqrt(2 * k)


def test_ga_step_is_deterministic_and_seeded(oracle_mod, prob):
    o = oracle_mod.Oracle(prob)
    g = _ga(pop=128)
    pop = o.ga_init(g, 5)
    fit = np.random.default_rng(0).standard_normal(128)
    a = o.ga_step(g, 5, 2, pop, fit)
    assert np.array_equal(a, o.ga_step(g, 5, 2, pop, fit))
    assert not np.array_equal(a, o.ga_step(g, 6, 2, pop, fit))
    assert not np.array_equal(a, o.ga_step(g, 5, 3, pop, fit))


def test_ga_finds_optimum_of_tiny_space(oracle_mod):
    """216 candidates, population 64 over 30 generations: the GA must reach the
    exhaustive optimum (the argmax over the same landscape, Sec. IV-C)."""
    p = W.tiny()
    o = oracle_mod.Oracle(p)
    ti, ts, _ = o.exhaustive(1)
    J, genome = o.ga_run(_ga(pop=64, gens=30), seed=1000)
    assert J == ts[0]
    assert list(genome) == list(o.decode(int(ti[0])))


@pytest.mark.parametrize("opts,seed,cap,coupled", [([12, 9, 9, 9, 9], 5, 30.0, False), ([5] * 8, 7, 45.0, False),
                                                  ([12, 9, 9, 9, 9], 5, 30.0, True), ([16] * 4, 6, 25.0, True)])
def test_integer_landscape_is_exact_in_any_order(oracle_mod, opts, seed, cap, coupled):
    """The premise of the bit-exact GA tests on the GPU: in the integer landscapes
    every input is an integer and the largest value any partial sum can reach is
    below 2**24, so fp32 arithmetic is exact whatever the summation order.  In the
    coupled variant the predictors also see the unscaled aggregate (summed demands
    and N), which stays an integer."""
    prob = W.integer_landscape(opts, seed, cap, objective="soft_lat", soft_penalty=0.5, coupled=coupled)
    n, d, h = len(opts), 8, 64
    per = W.param_count(d, h, h)
    for a in (prob["local_feats"], prob["demand"], prob["weights"], prob["sla"], prob["obj_w"]) + \
            ((prob["agg_scale"],) if coupled else ()):
        assert np.all(a == np.round(a))
    w = prob["weights"].reshape(n, per).astype(np.float64)
    x = float(np.abs(prob["local_feats"]).max())
    agg = np.append(n * np.abs(prob["demand"]).max(axis=0), n) * (prob["agg_scale"] if coupled else 0.0)
    b1 = h * (d + 4)
    for i in range(n):
        W1 = w[i, :b1].reshape(h, d + 4)
        assert np.any(W1[:, d:] != 0) if coupled else np.all(W1[:, d:] == 0)
        h1 = d * x * np.abs(W1[:, :d]).max() + float(np.abs(W1[:, d:]).max(axis=0) @ agg) + \
            np.abs(w[i, b1:b1 + h]).max()
        o2 = b1 + h
        h2 = h * h1 * np.abs(w[i, o2:o2 + h * h]).max() + np.abs(w[i, o2 + h * h:o2 + h * h + h]).max()
        o3 = o2 + h * h + h
        out = h * h2 * np.abs(w[i, o3:o3 + 2 * h]).max() + np.abs(w[i, o3 + 2 * h:]).max()
        bound_J = n * (float(prob["obj_w"].max()) * out + 0.5 * (out + float(np.abs(prob["sla"]).max())))
        assert bound_J < 2 ** 24
    o = oracle_mod.Oracle(prob)
    idx = np.random.default_rng(1).integers(0, o.space_size(), 3000).astype(np.uint64)
    s, f, pred, _ = o.score_list(idx, with_pred=True)
    assert np.all(pred == np.round(pred))
    assert f.any() and np.all(2 * s[f] == np.round(2 * s[f]))  # soft penalty 0.5: halves


# ---------------------------------------------------------------------------
# The GA loop (Sec. IV-C): which population is evaluated how often, and which
# individual is returned.  Each pin composes only separately pinned pieces (the
# initial population, the step operator, the predictor and objective).
# ---------------------------------------------------------------------------
def _fitness(o, pop):
    return np.array([o.score_digits(row)[0] for row in pop])


def test_ga_run_of_one_generation_returns_the_best_initial_individual(oracle_mod):
    """gens = 1 evaluates the initial population once and returns its fittest
    individual (lowest slot among equals), with no generation step."""
    p = W.random_small(21, 3, max_options=6, h1=16, vram_cap=30.0)
    o = oracle_mod.Oracle(p)
    for seed in (3, 4, 5):
        g = _ga(pop=48, gens=1)
        pop0 = o.ga_init(g, seed)
        fit = _fitness(o, pop0)
        e = int(np.argmax(fit))  # first maximum: the lowest slot among equals
        J, genome = o.ga_run(g, seed)
        assert J == fit[e]
        assert list(genome) == list(pop0[e])


@pytest.mark.parametrize("gens", [2, 3, 5])
def test_ga_run_is_the_initial_population_then_gens_minus_one_steps(oracle_mod, gens):
    """gens evaluations: the initial population, then a step with generation index
    0, 1, ..., gens - 2, each step taking the fitness of the population it breeds
    from; the result is the fittest individual of the last evaluated population."""
    p = W.random_small(22, 4, max_options=5, h1=16, vram_cap=40.0)
    o = oracle_mod.Oracle(p)
    g = _ga(pop=40, gens=gens)
    seed = 77
    pop = o.ga_init(g, seed)
    for gen in range(gens - 1):
        pop = o.ga_step(g, seed, gen, pop, _fitness(o, pop))
    fit = _fitness(o, pop)
    e = int(np.argmax(fit))
    J, genome = o.ga_run(g, seed)
    assert J == fit[e]
    assert list(genome) == list(pop[e])


def _two_option_problem(oracle_mod, seed):
    """One model with two options, both feasible (no SLA or VRAM limit in reach)."""
    p = W.make_problem([2], 8, 16, 0, seed, 1e9)
    p["sla"] = np.array([1e9], np.float32)
    o = oracle_mod.Oracle(p)
    J = [o.score_digits([k])[0] for k in (0, 1)]
    assert J[0] != J[1] and np.isfinite(J).all()
    return o, J


def test_ga_without_mutation_keeps_to_the_genes_of_the_initial_population(oracle_mod):
    """With mutation off, crossover and selection can only recombine genes already
    present: on one model with two options a population that starts without the
    better option never finds it, and one that starts with it returns it from the
    first generation on (elitism keeps it)."""
    o, J = _two_option_problem(oracle_mod, 31)
    best = int(np.argmax(J))
    seen = set()
    for seed in range(200):
        g = _ga(pop=2, gens=1, mutation_p=0.0, tournament=2)
        has_best = best in set(o.ga_init(g, seed)[:, 0].tolist())
        if has_best in seen:
            continue
        seen.add(has_best)
        expect = best if has_best else 1 - best  # two options: without the best, only the other
        for gens in range(1, 7):
            Jr, genome = o.ga_run(_ga(pop=2, gens=gens, mutation_p=0.0, tournament=2), seed)
            assert genome[0] == expect and Jr == J[expect]
        if len(seen) == 2:
            break
    assert seen == {True, False}


def test_ga_with_elitism_never_loses_its_best(oracle_mod):
    """One elite: the returned fitness does not decrease with the number of
    generations for a fixed seed."""
    p = W.random_small(23, 4, max_options=6, h1=16, vram_cap=35.0)
    o = oracle_mod.Oracle(p)
    Js = [o.ga_run(_ga(pop=24, gens=g), 9)[0] for g in range(1, 9)]
    assert all(b >= a for a, b in zip(Js, Js[1:]))
