"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Each test names what fixes the expected value: a number printed in the paper,
a value worked out by hand, a closed form, a library routine on a special case,
or brute force.  None of these runs on a GPU.
"""
import math

import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _O(oracle_mod, prob, **kw):
    return oracle_mod.Oracle(prob, **kw)


# ---------------------------------------------------------------------------
# Random-number generator: the published SplitMix64 sequence for state 0.
# ---------------------------------------------------------------------------

def test_splitmix64_published_outputs(oracle_mod):
    # Outputs 0..3 of SplitMix64 started from state 0 (Steele et al. 2014 /
    # Vigna's reference generator).
    ref = [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F, 0xF88BB8A8724C81EC]
    assert [oracle_mod.splitmix64(0, i) for i in range(4)] == ref


# ---------------------------------------------------------------------------
# Eq. 1: sizes of the joint space and the mixed-radix enumeration.
# ---------------------------------------------------------------------------

def _sized(ks):
    return W.make_problem(ks, 8, 32, 0, 7, 24.0)


def test_space_sizes_from_paper(oracle_mod):
    # Sec. III-A: the N = 2 space is 6 LLM x 27 vision = 162 configurations.
    assert _O(oracle_mod, _sized([6, 27])).space_size() == 162
    # Sec. IV-C / abstract: 78,732 joint configurations at N = 5
    # (two LLMs with 6 options, the AWQ-only 7B with 3, two YOLO11 with 27).
    assert _O(oracle_mod, _sized([6, 6, 3, 27, 27])).space_size() == 78732
    assert _O(oracle_mod, W.paper_scale()).space_size() == 78732
    assert _O(oracle_mod, W.tiny()).space_size() == 216
    assert _O(oracle_mod, W.large(precision="fp32")).space_size() == 24 ** 6
    assert _O(oracle_mod, W.stress(precision="fp32")).space_size() == 2 ** 32


def test_space_size_overflow_is_zero(oracle_mod):
    assert _O(oracle_mod, _sized([255] * 9)).space_size() == 0  # 255**9 > 2**64


@pytest.mark.parametrize("ks", [[12, 18], [6, 6, 3, 27, 27], [12, 9, 9, 9, 9], [3, 1, 7, 2]])
def test_decode_matches_numpy_unravel_index(oracle_mod, ks):
    o = _O(oracle_mod, _sized(ks))
    n = o.space_size()
    rs = np.random.default_rng(0)
    for idx in list(rs.integers(0, n, size=200)) + [0, n - 1]:
        assert list(o.decode(int(idx))) == list(np.unravel_index(int(idx), ks))


# ---------------------------------------------------------------------------
# Hand-worked two-model example (values computed by hand).
# ---------------------------------------------------------------------------

def test_hand_example_values(oracle_mod):
    o = _O(oracle_mod, W.hand_example())
    # idx 0 = (0, 0): A = (0.3, 10, 300, 2); h_A = 0.5 - 0.1 = 0.4 -> thr 0.8, lat 0.4;
    # h_B = relu(0.25 - 0.3) = 0 -> thr 0, lat 0; J = 0.8, feasible.
    J, f, pred, agg = o.score_digits([0, 0])
    assert f and J == pytest.approx(0.8, abs=1e-6)
    np.testing.assert_allclose(agg, [0.3, 10, 300, 2], rtol=1e-6)
    np.testing.assert_allclose(pred, [[0.8, 0.4], [0.0, 0.0]], atol=1e-6)
    # idx 1 = (0, 1): A = (0.5, 20, 500, 2); h_A = 0.3, h_B = 0.25; J = 0.6 + 0.25.
    J, f, pred, agg = o.score_digits([0, 1])
    assert f and J == pytest.approx(0.85, abs=1e-6)
    np.testing.assert_allclose(pred, [[0.6, 0.3], [0.25, 0.5]], atol=1e-6)
    # idx 2 = (1, 0): h_A = 1.0 - 0.16 = 0.84 > SLA 0.8 -> infeasible.
    J, f, pred, _ = o.score_digits([1, 0])
    assert not f and J == -math.inf and pred[0, 1] == pytest.approx(0.84, abs=1e-6)
    # idx 3 = (1, 1): Sigma VRAM = 26 > 24 -> infeasible.
    J, f, _, agg = o.score_digits([1, 1])
    assert not f and J == -math.inf and agg[1] == pytest.approx(26.0)
    ti, ts, cnt = o.exhaustive(2)
    assert cnt == 2 and list(ti) == [1, 0]
    np.testing.assert_allclose(ts, [0.85, 0.8], atol=1e-6)


def test_hand_example_soft_latency_objective(oracle_mod):
    p = W.hand_example()
    p["objective"], p["soft_penalty"] = "soft_lat", 0.1
    o = _O(oracle_mod, p)
    # Soft mode: only VRAM is a hard constraint.  idx 2: thr = 1.68 + 0,
    # latency excess 0.84 - 0.8 = 0.04 -> J = 1.68 - 0.1 * 0.04 = 1.676.
    J, f, _, _ = o.score_digits([1, 0])
    assert f and J == pytest.approx(1.676, abs=1e-6)
    J, f, _, _ = o.score_digits([1, 1])
    assert not f  # VRAM 26 > 24 stays infeasible
    ti, ts, cnt = o.exhaustive(3)
    assert cnt == 3 and list(ti) == [2, 1, 0]


def test_hand_example_no_feasible(oracle_mod):
    p = W.hand_example()
    p["vram_cap"] = 1.0
    ti, ts, cnt = _O(oracle_mod, p).exhaustive(3)
    assert cnt == 0 and all(int(i) == 2 ** 64 - 1 for i in ti) and all(s == -math.inf for s in ts)


# ---------------------------------------------------------------------------
# Special cases that reduce to library routines or closed forms.
# ---------------------------------------------------------------------------

def _unpack(prob, i):
    dl, h1, h2 = prob["d_local"], prob["hidden1"], prob["hidden2"]
    din = dl + 4
    w = prob["weights"].astype(np.float64)
    per = W.param_count(dl, h1, h2)
    w = w[i * per:(i + 1) * per]
    o = 0
    W1 = w[o:o + h1 * din].reshape(h1, din); o += h1 * din
    b1 = w[o:o + h1]; o += h1
    layers = [(W1, b1)]
    last = h1
    if h2:
        W2 = w[o:o + h2 * h1].reshape(h2, h1); o += h2 * h1
        b2 = w[o:o + h2]; o += h2
        layers.append((W2, b2))
        last = h2
    W3 = w[o:o + 2 * last].reshape(2, last); o += 2 * last
    b3 = w[o:o + 2]
    layers.append((W3, b3))
    return layers


@pytest.mark.parametrize("shape", [(8, 32, 16), (8, 32, 0), (16, 24, 40)])
def test_linear_case_is_one_affine_map(oracle_mod, shape):
    """With non-negative weights and inputs every ReLU is the identity, so each
    predictor collapses to the affine map z -> M z + c with M = W3 W2 W1
    (composed with numpy matmul, not layer by layer)."""
    dl, h1, h2 = shape
    prob = W.make_problem([3, 4, 5], dl, h1, h2, seed=11, vram_cap=1e9)
    prob["weights"] = np.abs(prob["weights"])
    o = _O(oracle_mod, prob)
    offs = np.concatenate([[0], np.cumsum(prob["n_options"])])
    for idx in range(0, o.space_size(), 7):
        digits = o.decode(idx)
        _, _, pred, agg = o.score_digits(digits)
        rows = offs[:-1] + digits
        A = prob["demand"][rows].astype(np.float64).sum(axis=0)
        a = np.concatenate([A, [len(digits)]]) * prob["agg_scale"].astype(np.float64)
        for i in range(len(digits)):
            layers = _unpack(prob, i)
            M = np.eye(layers[0][0].shape[1])
            c = np.zeros(layers[0][0].shape[1])
            for Wl, bl in layers:
                M, c = Wl @ M, Wl @ c + bl
            z = np.concatenate([prob["local_feats"][rows[i]].astype(np.float64), a])
            np.testing.assert_allclose(pred[i], M @ z + c, rtol=1e-12, atol=1e-12)


def test_aggregate_is_sum_of_demand_rows(oracle_mod):
    prob = W.paper_scale()
    o = _O(oracle_mod, prob)
    offs = np.concatenate([[0], np.cumsum(prob["n_options"])])
    rs = np.random.default_rng(1)
    idx = rs.integers(0, o.space_size(), size=300).astype(np.uint64)
    _, _, _, agg = o.score_list(idx, with_pred=True)
    digits = np.stack(np.unravel_index(idx.astype(np.int64), prob["n_options"]), axis=1)
    rows = offs[:-1][None, :] + digits
    dem = prob["demand"].astype(np.float64)[rows]              # [n, N, 3]
    np.testing.assert_array_equal(agg[:, :3], dem.sum(axis=1))  # exact in fp64
    np.testing.assert_array_equal(agg[:, 3], 5.0)


def _separable(prob):
    """Zero every aggregate column of W1 so model i depends on its own option only."""
    prob = dict(prob)
    dl, h1, h2 = prob["d_local"], prob["hidden1"], prob["hidden2"]
    din, per = dl + 4, W.param_count(dl, h1, h2)
    w = prob["weights"].copy()
    for i in range(prob["n_options"].size):
        W1 = w[i * per:i * per + h1 * din].reshape(h1, din)
        W1[:, dl:] = 0.0
    prob["weights"] = w
    prob["vram_cap"] = 1e30
    return prob


@pytest.mark.parametrize("sla_range", [(0.5, 2.0), W.TIGHT_SLA])
def test_separable_closed_form(oracle_mod, sla_range):
    """Separable case: argmax = per-model argmax of w_i thr_i over the options
    meeting SLA_i; feasible count = prod_i #{o : lat_i(o) <= SLA_i}."""
    prob = _separable(W.paper_scale())
    W.set_scenario(prob, 77, sla_range)
    o = _O(oracle_mod, prob)
    ks = prob["n_options"]
    best_digits, count = [], 1
    for i, k in enumerate(ks):
        vals = []
        for opt in range(k):
            d = [0] * len(ks)
            d[i] = opt
            _, _, pred, _ = o.score_digits(d)
            vals.append(pred[i])
        vals = np.array(vals)
        ok = vals[:, 1] <= float(prob["sla"][i])
        count *= int(ok.sum())
        if ok.any():
            cand = np.where(ok, float(prob["obj_w"][i]) * vals[:, 0], -np.inf)
            best_digits.append(int(np.argmax(cand)))
    ti, ts, cnt = o.exhaustive(4)
    assert cnt == count
    if count:
        assert list(o.decode(int(ti[0]))) == best_digits


def test_vram_only_count_two_pointer(oracle_mod):
    """With SLA = +inf the count is #{(a, b): v_a + v_b <= C}; counted with a sort
    and a two-pointer sweep."""
    prob = W.tiny()
    prob["sla"] = np.full(2, 1e30, dtype=np.float32)
    o = _O(oracle_mod, prob)
    v = prob["demand"][:, 1].astype(np.float64)
    va, vb = np.sort(v[:12]), np.sort(v[12:])
    C, j, cnt = prob["vram_cap"], len(vb) - 1, 0
    for x in va:
        while j >= 0 and x + vb[j] > C:
            j -= 1
        cnt += j + 1
    _, _, c = o.exhaustive(8)
    assert c == cnt and 0 < cnt < 216


def test_sigmoid_head_closed_form(oracle_mod):
    p = W.hand_example()
    p["out_act"] = "sigmoid"
    w = p["weights"].copy()
    for i in range(2):  # W3 = 0, b3 = (0, ln 3): thr = 1/2, lat = 3/4 for every option
        w[i * 12 + 8:i * 12 + 12] = [0, 0, 0, math.log(3.0)]
    p["weights"] = w
    p["sla"] = np.array([0.8, 0.8], dtype=np.float32)
    o = _O(oracle_mod, p)
    J, f, pred, _ = o.score_digits([0, 0])
    assert f and J == pytest.approx(1.0, abs=1e-7)
    np.testing.assert_allclose(pred, [[0.5, 0.75], [0.5, 0.75]], atol=1e-7)
    p["sla"] = np.array([0.8, 0.7], dtype=np.float32)
    assert _O(oracle_mod, p).exhaustive(2)[2] == 0  # 0.75 > 0.7 everywhere


@pytest.mark.parametrize("pos", ["W1", "b3"])
def test_nan_weights_make_candidates_infeasible(oracle_mod, pos):
    """A NaN weight of model 0 reaches its outputs (ReLU keeps NaN), so J is NaN
    and every candidate is infeasible."""
    p = W.tiny()
    p["weights"] = p["weights"].copy()
    per = W.param_count(8, 32, 0)
    p["weights"][0 if pos == "W1" else per - 1] = np.nan
    _, _, cnt = _O(oracle_mod, p).exhaustive(4)
    assert cnt == 0


# ---------------------------------------------------------------------------
# Invariants and brute force.
# ---------------------------------------------------------------------------

def _brute_topk(o, k):
    n = o.space_size()
    idx = np.arange(n, dtype=np.uint64)
    s, f = o.score_list(idx)
    order = np.lexsort((idx, -s))  # J descending, index ascending
    keep = [int(i) for i in order if f[i]][:k]
    return keep, s, int(f.sum())


@pytest.mark.parametrize("seed", [1, 2, 3, 4, 5])
def test_exhaustive_equals_brute_force(oracle_mod, seed):
    prob = W.random_small(seed, n_models=4, max_options=7, h2=16, vram_cap=35.0,
                          sla_range=(0.3, 1.0))
    o = _O(oracle_mod, prob)
    k = 10
    keep, s, cnt = _brute_topk(o, k)
    for nt in (1, 8):
        ti, ts, c = o.exhaustive(k, nthreads=nt)
        assert c == cnt
        assert [int(i) for i in ti[:len(keep)]] == keep
        np.testing.assert_array_equal(ts[:len(keep)], s[keep])


def test_ties_ordered_by_index(oracle_mod):
    prob = W.make_problem([4, 5], 8, 16, 0, 3, 1e9)
    prob["local_feats"][:] = 0.5
    prob["demand"][:] = [0.1, 1.0, 100.0]
    prob["sla"][:] = 1e30
    o = _O(oracle_mod, prob)
    ti, ts, cnt = o.exhaustive(7)
    assert cnt == 20 and list(ti) == list(range(7)) and np.all(ts == ts[0])


def test_candidate_order_invariance(oracle_mod):
    prob = W.paper_scale()
    W.set_scenario(prob, 5, (0.4, 0.9))
    o = _O(oracle_mod, prob)
    rs = np.random.default_rng(3)
    idx = rs.integers(0, o.space_size(), size=500).astype(np.uint64)
    perm = rs.permutation(idx.size)
    s1, f1 = o.score_list(idx)
    s2, f2 = o.score_list(idx[perm])
    np.testing.assert_array_equal(s1[perm], s2)
    np.testing.assert_array_equal(f1[perm], f2)


def test_model_permutation_permutes_argmax(oracle_mod):
    prob = W.random_small(9, n_models=3, max_options=6, h2=8, vram_cap=30.0)
    o = _O(oracle_mod, prob)
    perm = [2, 0, 1]
    ks = prob["n_options"]
    offs = np.concatenate([[0], np.cumsum(ks)])
    per = W.param_count(prob["d_local"], prob["hidden1"], prob["hidden2"])
    q = dict(prob)
    q["n_options"] = ks[perm]
    q["local_feats"] = np.concatenate([prob["local_feats"][offs[i]:offs[i + 1]] for i in perm])
    q["demand"] = np.concatenate([prob["demand"][offs[i]:offs[i + 1]] for i in perm])
    q["weights"] = np.concatenate([prob["weights"][i * per:(i + 1) * per] for i in perm])
    q["sla"], q["obj_w"] = prob["sla"][perm], prob["obj_w"][perm]
    oq = _O(oracle_mod, q)
    ti, ts, c = o.exhaustive(1)
    tq, tsq, cq = oq.exhaustive(1)
    assert c == cq and ts[0] == pytest.approx(tsq[0], rel=1e-12)
    assert list(o.decode(int(ti[0]))[perm]) == list(oq.decode(int(tq[0])))


def test_default_agg_scale(oracle_mod):
    prob = W.paper_scale()
    ref = _O(oracle_mod, prob).score_list(np.arange(50, dtype=np.uint64))[0]
    prob = dict(prob)
    prob["agg_scale"] = None
    got = _O(oracle_mod, prob).score_list(np.arange(50, dtype=np.uint64))[0]
    np.testing.assert_array_equal(ref, got)


def test_pred_scale_equals_output_in_linear_case(oracle_mod):
    """With non-negative weights and inputs no term of the final dot product
    cancels, so the condition scale equals |output|."""
    prob = W.make_problem([3, 4], 8, 16, 8, 11, 1e9)
    prob["weights"] = np.abs(prob["weights"])
    o = _O(oracle_mod, prob)
    idx = np.arange(o.space_size(), dtype=np.uint64)
    _, _, pred, _ = o.score_list(idx, with_pred=True)
    np.testing.assert_allclose(o.pred_scale(idx), np.abs(pred), rtol=1e-12)


def test_pred_scale_hand_value(oracle_mod):
    """One input x = 0.5, two hidden units h = (x, 0.5 x) = (0.5, 0.25), throughput
    row W3 = (1, -1): thr = 0.25 while the terms have magnitude 0.5 + 0.25 = 0.75."""
    p = dict(n_options=np.array([1], np.int32), d_local=1, hidden1=2, hidden2=0,
             local_feats=np.array([[0.5]], np.float32), demand=np.array([[0.1, 1.0, 10.0]], np.float32),
             weights=np.array([1, 0, 0, 0, 0, 0.5, 0, 0, 0, 0,  0, 0,  1, -1, 0, 0,  0, 0], np.float32),
             agg_scale=np.ones(4, np.float32), sla=np.array([9.0], np.float32),
             obj_w=np.ones(1, np.float32), vram_cap=100.0)
    o = _O(oracle_mod, p)
    J, f, pred, _ = o.score_digits([0])
    assert pred[0, 0] == pytest.approx(0.25)
    np.testing.assert_allclose(o.pred_scale(np.array([0], np.uint64))[0, 0], [0.75, 0.0], atol=1e-12)


def _feasible_fraction(oracle_mod, prob, sample=40000):
    o = _O(oracle_mod, prob)
    n = o.space_size()
    idx = np.arange(n, dtype=np.uint64) if n <= sample else \
        np.random.default_rng(0).integers(0, n, sample).astype(np.uint64)
    return float(o.score_list(idx)[1].mean())


def test_scenarios_that_exercise_the_masks_bind_on_part_of_the_space(oracle_mod):
    """The parity tests' and the benchmark's mask scenarios leave a feasible fraction
    strictly between 0 and 1: a mask that rejects everything (or nothing) would let a
    wrong feasibility test pass unnoticed."""
    import test_gpu_parity as tp
    import test_gpu_tc as tt
    cases = {"parity." + k: tp.PROBLEMS[k] for k in ("tight", "odd_shape", "sigmoid")}
    cases.update({"tc." + k: tt.PROBLEMS[k] for k in ("tight", "odd", "p6432", "multipass")})
    for seed in (1, 2, 3, 4, 5):
        cases[f"brute{seed}"] = W.random_small(seed, n_models=4, max_options=7, h2=16, vram_cap=35.0,
                                               sla_range=(0.3, 1.0))
    cases["order"] = W.set_scenario(W.paper_scale(), 5, (0.4, 0.9))
    cases["set_objective"] = W.set_scenario(W.paper_scale(), 123, (-0.1, 0.8))
    large = W.large(precision="fp32")
    cases["bench_tight"] = W.set_scenario(large, 31, W.TIGHT_SLA)
    for name, prob in cases.items():
        fr = _feasible_fraction(oracle_mod, prob)
        assert 0.0 < fr < 1.0, (name, fr)
