"""Pins of the oracle's fixed-context mode (Sec. III-B: the observed state s_t is
held fixed during the search; Eq. 3 utility; Eq. 4 constraints; Lambda built
without its VRAM-infeasible configurations)."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W


def _hand_fc():
    """The two-model hand example under an observed state (0.5 SM, 20 GB, 300 GB/s, N=2).

    Model A: fhat = 2 relu(x - 0.01 VRAM) -> options x = 0.5, 1.0 give fhat = 0.6, 1.6;
    with f_min = 0, f_max = 2: f = 0.3, 0.8.  Model B: fhat = relu(x - SM) -> x = 0.25,
    0.75 give f = 0, 0.25 (f_max = 1).  Floors tau = (0.2, 0.1): B's option 0 fails.
    Variants (0, 1) per model, A in use with variant 0, B none; Q = (1.000, 0.979) for A,
    (0.73, 0.96) for B; c = (30, 5); alpha = 1/60, beta = 5, delta = 0.05:
      u_A(0) = 0.3 * 1.000                       = 0.3
      u_A(1) = 0.8 * 0.979 - 30 / 60             = 0.2832   (reload of A)
      u_B(0) = 0 - 5 * (0.1 + 0.05 - 0)^2        = -0.1125  (below its floor anyway)
      u_B(1) = 0.25 * 0.96 - 5 * max(0, 0.15 - 0.25)^2 = 0.24
    Joint: (0,0) B floor fails; (0,1) J = 0.54, VRAM 4 + 16 = 20 <= 24; (1,0) floor;
    (1,1) VRAM 26 > 24.  Best idx 1, J = 0.54, feasible count 1."""
    return dict(obs=np.array([0.5, 20.0, 300.0, 2.0], np.float32),
                variant=np.array([0, 1, 0, 1], np.int32),
                quality=np.array([1.0, 0.979, 0.73, 0.96], np.float32),
                f_min=np.zeros(4, np.float32), f_max=np.array([2.0, 2.0, 1.0, 1.0], np.float32),
                omega=np.ones(2, np.float32), tau=np.array([0.2, 0.1], np.float32),
                reload_cost=np.array([30.0, 5.0], np.float32), prev_variant=np.array([0, -1], np.int32),
                alpha=1.0 / 60.0, beta=5.0, delta=0.05)


def test_fc_hand_example(oracle_mod):
    o = oracle_mod.Oracle(W.hand_example())
    fc = _hand_fc()
    fhat, f, ok, u = o.fc_local(fc)
    np.testing.assert_allclose(fhat, [0.6, 1.6, 0.0, 0.25], atol=1e-6)
    np.testing.assert_allclose(f, [0.3, 0.8, 0.0, 0.25], atol=1e-6)
    assert list(ok) == [True, True, False, True]
    np.testing.assert_allclose(u, [0.3, 0.2832, -0.1125, 0.24], atol=1e-6)
    ti, ts, cnt = o.fc_exhaustive(fc, 4)
    assert cnt == 1 and int(ti[0]) == 1 and abs(ts[0] - 0.54) < 1e-6
    assert all(int(i) == 2 ** 64 - 1 for i in ti[1:]) and np.all(np.isneginf(ts[1:]))
    for d, (J, feas) in {(0, 0): (-np.inf, False), (1, 0): (-np.inf, False), (1, 1): (-np.inf, False)}.items():
        assert o.fc_score_digits(fc, d) == (J, feas)


def test_fc_separable_closed_form(oracle_mod):
    """With the VRAM bound slack, J(lambda) = sum_i u_i(o_i) over floor-feasible
    options: the argmax is the per-model argmax of u, and the count is the product of
    the per-model numbers of floor-feasible options."""
    prob = W.paper_scale()
    prob["vram_cap"] = 1e9
    fc = W.fc_scenario(prob, 3)
    o = oracle_mod.Oracle(prob)
    _, _, ok, u = o.fc_local(fc)
    off = np.concatenate([[0], np.cumsum(prob["n_options"])])
    best, count, Jbest = [], 1, 0.0
    for i in range(len(prob["n_options"])):
        ui = np.where(ok[off[i]:off[i + 1]], u[off[i]:off[i + 1]], -np.inf)
        best.append(int(np.argmax(ui)))
        Jbest += float(np.max(ui))
        count *= int(ok[off[i]:off[i + 1]].sum())
    assert 0 < count < o.space_size()
    ti, ts, cnt = o.fc_exhaustive(fc, 1)
    assert cnt == count
    assert list(o.decode(int(ti[0]))) == best
    assert abs(ts[0] - Jbest) <= 1e-12 * max(1.0, abs(Jbest))


def test_fc_reload_term_is_alpha_c(oracle_mod):
    """Switching the variant in use of one model changes J of a configuration that
    keeps (resp. leaves) that variant by exactly -alpha c_i (resp. +alpha c_i)."""
    prob = W.paper_scale()
    prob["vram_cap"] = 1e9
    fc = W.fc_scenario(prob, 6)
    o = oracle_mod.Oracle(prob)
    ti, ts, _ = o.fc_exhaustive(fc, 1)
    d = o.decode(int(ti[0]))
    row = int(d[1]) + int(prob["n_options"][0])  # model 1's chosen option row
    v = int(fc["variant"][row])
    same, other = dict(fc), dict(fc)
    same["prev_variant"] = fc["prev_variant"].copy(); same["prev_variant"][1] = v
    other["prev_variant"] = fc["prev_variant"].copy(); other["prev_variant"][1] = v + 1
    Js, _ = o.fc_score_digits(same, d)
    Jo, _ = o.fc_score_digits(other, d)
    ac = float(np.float32(fc["alpha"])) * float(fc["reload_cost"][1])
    assert abs((Js - Jo) - ac) <= 1e-12


def test_fc_margin_penalty_is_quadratic_below_the_margin(oracle_mod):
    """u(beta) - u(0) = -beta max(0, tau_i + delta - f)^2 for every option: zero at and
    above the margin, quadratic below (compared over beta = 0, 5, 10)."""
    prob = W.paper_scale()
    fc = W.fc_scenario(prob, 4)
    o = oracle_mod.Oracle(prob)
    us = []
    for beta in (0.0, 5.0, 10.0):
        _, f, _, u = o.fc_local(dict(fc, beta=beta))
        us.append(u)
    d5, d10 = us[0] - us[1], us[0] - us[2]
    np.testing.assert_allclose(d10, 2 * d5, rtol=1e-12, atol=1e-15)
    assert np.all(d5 >= 0)
    tau = np.repeat(fc["tau"], prob["n_options"]).astype(np.float64)
    margin = tau + float(np.float32(fc["delta"])) - f
    assert np.all(d5[margin <= 0] == 0) and np.all(d5[margin > 0] > 0)
    np.testing.assert_allclose(d5[margin > 0], 5.0 * margin[margin > 0] ** 2, rtol=1e-9)


def test_fc_linear_case_is_one_matrix_product(oracle_mod):
    """Nonnegative weights and inputs: every ReLU passes its input, so fhat is the
    product of the layer matrices applied to [x | obs * s_A]; with f_min = 0,
    f_max = 1, Q = 1, alpha = beta = 0: u = omega fhat."""
    prob = W.make_problem([3, 4], 8, 16, 8, 5, 1e9)
    w = np.abs(prob["weights"])
    prob["weights"] = w
    n, rows = 2, 7
    fc = dict(W.fc_scenario(prob, 2), f_min=np.zeros(rows, np.float32), f_max=np.ones(rows, np.float32),
              quality=np.ones(rows, np.float32), alpha=0.0, beta=0.0,
              omega=np.array([1.5, 0.5], np.float32))
    o = oracle_mod.Oracle(prob)
    fhat, _, _, u = o.fc_local(fc)
    per = W.param_count(8, 16, 8)
    zs = fc["obs"].astype(np.float64) * prob["agg_scale"].astype(np.float64)
    off = [0, 3, 7]
    for i in range(n):
        p = w[i * per:(i + 1) * per].astype(np.float64)
        W1 = p[:16 * 12].reshape(16, 12); b1 = p[192:208]
        W2 = p[208:208 + 128].reshape(8, 16); b2 = p[336:344]
        W3 = p[344:360].reshape(2, 8); b3 = p[360:362]
        X = np.hstack([prob["local_feats"][off[i]:off[i + 1]].astype(np.float64),
                       np.tile(zs, (off[i + 1] - off[i], 1))])
        want = ((X @ W1.T + b1) @ W2.T + b2) @ W3.T + b3
        np.testing.assert_allclose(fhat[off[i]:off[i + 1]], want[:, 0], rtol=1e-12)
        np.testing.assert_allclose(u[off[i]:off[i + 1]], fc["omega"][i] * want[:, 0], rtol=1e-6)


def test_vram_feasible_list_matches_two_pointer_count(oracle_mod):
    """Lambda without its VRAM-infeasible configurations (Eq. 4 applied while building
    Lambda): the count equals a sort + two-pointer count of pairs with vram_a + vram_b
    <= R, and the list is exactly the ascending indices that satisfy the bound."""
    prob = W.tiny()
    o = oracle_mod.Oracle(prob)
    c, lst = o.vram_feasible()
    va = np.sort(prob["demand"][:12, 1].astype(np.float64))
    vb = np.sort(prob["demand"][12:, 1].astype(np.float64))
    cap = float(prob["vram_cap"])
    j, want = len(vb), 0
    for a in va:
        while j > 0 and a + vb[j - 1] > cap:
            j -= 1
        want += j
    assert c == want and 0 < c < 216
    idx = np.arange(216)
    ok = (prob["demand"][idx // 18, 1].astype(np.float64) + prob["demand"][12 + idx % 18, 1].astype(np.float64)) <= cap
    assert np.array_equal(lst, idx[ok].astype(np.uint64))
    c2, lst2 = o.vram_feasible(50, 150, cap=10)
    assert c2 == int(ok[50:150].sum()) and np.array_equal(lst2, idx[50:150][ok[50:150]][:10].astype(np.uint64))


# ---------------------------------------------------------------------------
# The Eq. 3 utility on the coupled aggregate (the predictors see the candidate's
# own summed demands)
# ---------------------------------------------------------------------------

def test_util_hand_example(oracle_mod):
    """The hand example's coupled aggregate of (0, 1) is (0.5 SM, 20 GB, ...), the
    observed state of the fixed-context hand example, so J(1) = 0.54 again; (0, 0)
    (aggregate 0.3 SM, 10 GB) and (1, 0) (0.5 SM, 16 GB) leave model B at f = 0 below
    its floor, (1, 1) exceeds 24 GB."""
    o = oracle_mod.Oracle(W.hand_example())
    fc = _hand_fc()
    J, f, pred = o.util_score_digits(fc, [0, 1])
    assert f and abs(J - 0.54) < 1e-6
    np.testing.assert_allclose(pred[:, 0], [0.6, 0.25], atol=1e-6)
    J0, f0, p0 = o.util_score_digits(fc, [0, 0])
    assert not f0 and J0 == -np.inf
    np.testing.assert_allclose(p0[:, 0], [0.8, 0.0], atol=1e-6)  # A: 2 relu(0.5 - 0.1), B: relu(0.25 - 0.3)
    J2, f2, p2 = o.util_score_digits(fc, [1, 0])
    assert not f2 and abs(p2[0, 0] - 1.68) < 1e-6
    ti, ts, cnt = o.util_exhaustive(fc, 4)
    assert cnt == 1 and int(ti[0]) == 1 and abs(ts[0] - 0.54) < 1e-6


def test_util_equals_fixed_context_when_the_aggregate_is_unused(oracle_mod):
    """With W1's aggregate columns zero, the coupled utility cannot see the aggregate,
    so it equals the fixed-context utility under any observed state."""
    prob = W.make_problem([4, 3, 5], 8, 32, 16, 9, 30.0)
    per = W.param_count(8, 32, 16)
    w = prob["weights"].copy()
    for i in range(3):
        W1 = w[i * per:i * per + 32 * 12].reshape(32, 12)
        W1[:, 8:] = 0.0
    prob["weights"] = w
    fc = W.fc_scenario(prob, 6)
    o = oracle_mod.Oracle(prob)
    for obs in (fc["obs"], np.array([9.0, 1.0, 123.0, 3.0], np.float32)):
        f2 = dict(fc, obs=obs)
        a = o.util_exhaustive(f2, 16)
        b = o.fc_exhaustive(f2, 16)
        assert a[2] == b[2] and 0 < a[2] < o.space_size()
        assert np.array_equal(a[0], b[0])
        np.testing.assert_allclose(a[1], b[1], rtol=1e-12)


def test_util_reduces_to_weighted_throughput(oracle_mod):
    """f_min = 0, f_max = 1, Q = 1, alpha = beta = 0, omega = w and floors far below:
    J = sum_i w_i thr_i, the weighted-throughput objective with the SLA switched off."""
    prob = W.paper_scale()
    rows = int(prob["n_options"].sum())
    fc = dict(W.fc_scenario(prob, 3), f_min=np.zeros(rows, np.float32), f_max=np.ones(rows, np.float32),
              quality=np.ones(rows, np.float32), alpha=0.0, beta=0.0, omega=prob["obj_w"],
              tau=np.full(5, -1e30, np.float32))
    ref = dict(prob, sla=np.full(5, 1e30, np.float32))
    o, r = oracle_mod.Oracle(prob), oracle_mod.Oracle(ref)
    idx = np.random.default_rng(2).integers(0, o.space_size(), 500).astype(np.uint64)
    a, fa = o.util_score_list(fc, idx)
    b, fb = r.score_list(idx)
    assert np.array_equal(fa, fb) and fa.all()
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-15)


# ---------------------------------------------------------------------------
# The paper's GA on the fixed-context landscape
# ---------------------------------------------------------------------------

def test_paper_ga_finds_the_optimum_of_the_paper_space(oracle_mod):
    """Pop 100, 30 generations (Sec. IV-C) on the 78,732-configuration space: the
    decision is within 0.5 % of the exhaustive optimum for every seed tried (the paper
    reports 0.10 % average, 0.38 % worst gap)."""
    prob = W.paper_scale()
    o = oracle_mod.Oracle(prob)
    for sc in (3, 6):
        fc = W.fc_scenario(prob, sc)
        _, ts, _ = o.fc_exhaustive(fc, 1)
        for seed in (1000, 1001, 1002):
            J, g = o.fc_ga_run(fc, W.PAPER_GA_PARAMS, seed)
            assert o.fc_score_digits(fc, g) == (J, True)
            assert J >= ts[0] - 0.005 * abs(ts[0])


def test_paper_ga_repair_reaches_a_feasible_decision(oracle_mod):
    """High floors leave a small feasible set: without repair the random population
    holds no feasible individual and the decision is infeasible; with repair
    (rejection sampling) it is feasible."""
    prob = W.paper_scale()
    o = oracle_mod.Oracle(prob)
    fc = W.fc_scenario(prob, 3)
    _, f, _, _ = o.fc_local(fc)
    off = np.concatenate([[0], np.cumsum(prob["n_options"])])
    # each model's floor just below its second-best normalised throughput: 2 feasible options per model
    tau = np.array([np.sort(f[off[i]:off[i + 1]])[-2] - 1e-6 for i in range(5)], np.float32)
    hard = dict(fc, tau=tau)
    _, _, cnt = o.fc_exhaustive(hard, 1)
    assert 0 < cnt <= 32
    g0 = dict(W.PAPER_GA_PARAMS, repair=0, mutation_p=0.0, gens=2)
    J0, _ = o.fc_ga_run(hard, g0, 5)
    assert J0 == -np.inf
    J1, g1 = o.fc_ga_run(hard, dict(W.PAPER_GA_PARAMS, gens=2), 5)
    assert np.isfinite(J1) and o.fc_score_digits(hard, g1)[1]


def test_paper_ga_is_deterministic_and_seeded(oracle_mod):
    prob = W.paper_scale()
    o = oracle_mod.Oracle(prob)
    fc = W.fc_scenario(prob, 6)
    g = dict(W.PAPER_GA_PARAMS, gens=3)
    a = o.fc_ga_run(fc, g, 11)
    assert a[0] == o.fc_ga_run(fc, g, 11)[0] and np.array_equal(a[1], o.fc_ga_run(fc, g, 11)[1])
    outs = {tuple(o.fc_ga_run(fc, g, s)[1]) for s in range(11, 19)}
    assert len(outs) > 1  # three generations do not always reach the same configuration


# ---------------------------------------------------------------------------
# The paper GA's loop (Sec. IV-C), pinned by pieces that have their own pins:
# the counter-based generator (published SplitMix64 outputs), the integer draw
# rule (multiply-shift of the top 32 bits) and the fixed-context table.
# ---------------------------------------------------------------------------
def _all_feasible_fc(prob, seed):
    fc = W.fc_scenario(prob, seed)
    return dict(fc, tau=np.full(len(prob["n_options"]), -1e6, np.float32))


def test_paper_ga_of_one_generation_returns_the_best_initial_draw(oracle_mod):
    """gens = 1: the initial population alone, individual c drawing gene i as
    floor(hi32(rng(seed, 0, c, init, i)) * K_i / 2^32); without repair and with no
    floor or VRAM limit in reach the result is the individual with the largest
    sum of table utilities (lowest slot among equals)."""
    prob = W.paper_scale()
    prob = dict(prob, vram_cap=1e9)
    o = oracle_mod.Oracle(prob)
    fc = _all_feasible_fc(prob, 4)
    _, _, ok, u = o.fc_local(fc)
    assert ok.all()
    K = [int(k) for k in prob["n_options"]]
    off = np.concatenate([[0], np.cumsum(K)])
    g = dict(W.PAPER_GA_PARAMS, gens=1, repair=0, pop=37)
    for seed in (1000, 1001):
        pop = np.array([[((oracle_mod.rng(seed, 0, c, 0, i) >> 32) * K[i]) >> 32 for i in range(len(K))]
                        for c in range(g["pop"])])
        fit = np.array([sum(u[off[i] + pop[c, i]] for i in range(len(K))) for c in range(g["pop"])])
        e = int(np.argmax(fit))
        J, genome = o.fc_ga_run(fc, g, seed)
        assert list(genome) == list(pop[e])
        assert J == pytest.approx(fit[e], rel=0, abs=1e-12)


def test_paper_ga_without_mutation_or_crossover_keeps_the_initial_genes(oracle_mod):
    """p_m = 0 and p_c = 0: every child copies a tournament winner, so on one model
    with two options the decision over any number of generations is the best option
    present in the initial population."""
    prob = W.make_problem([2], 8, 16, 0, 41, 1e9)
    o = oracle_mod.Oracle(prob)
    fc = _all_feasible_fc(prob, 41)
    _, _, ok, u = o.fc_local(fc)
    assert ok.all() and u[0] != u[1]
    seen = set()
    for seed in range(300):
        g0 = dict(W.PAPER_GA_PARAMS, pop=2, gens=1, repair=0, mutation_p=0.0, crossover_p=0.0)
        init = [((oracle_mod.rng(seed, 0, c, 0, 0) >> 32) * 2) >> 32 for c in range(2)]
        kind = tuple(sorted(set(init)))
        if kind in seen:
            continue
        seen.add(kind)
        expect = max(kind, key=lambda k: u[k])
        for gens in range(1, 7):
            J, genome = o.fc_ga_run(fc, dict(g0, gens=gens), seed)
            assert genome[0] == expect and J == pytest.approx(u[expect], rel=0, abs=1e-12)
        if len(seen) == 3:
            break
    assert seen == {(0,), (1,), (0, 1)}
