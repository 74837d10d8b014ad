"""Fixed-context mode on the GPU (mf_fc_set / mf_fc_table / mf_fc_search /
mf_vram_feasible) against the oracle: the per-option table element by element, the
search's count, best and top-k, the VRAM-feasible list bit for bit, and at full size
the closed form the fixed context gives (with the VRAM bound slack, J separates
into one term per model)."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

from test_oracle_fc import _hand_fc

pytestmark = pytest.mark.gpu

RTOL = 1e-5
NEAR = 1e-4


@pytest.fixture(scope="module")
def mf():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_02109_gb300 import build
    build.build()
    from paper_2609_02109_gb300 import mf as mod
    return mod


def _cases():
    tight = W.paper_scale()
    tight["vram_cap"] = 55.0  # binds: five options of 1-20 GB
    sig = W.random_small(21, n_models=4, max_options=8, h2=32, vram_cap=40.0, out_act="sigmoid")
    sixteen = W.make_problem([2] * 16, 8, 32, 32, 33, 180.0)
    return {
        "hand": (W.hand_example(), _hand_fc()),
        "tiny": (W.tiny(), W.fc_scenario(W.tiny(), 4)),
        "paper": (W.paper_scale(), W.fc_scenario(W.paper_scale(), 3)),
        "paper_vram_binds": (tight, W.fc_scenario(tight, 6)),
        "sigmoid": (sig, W.fc_scenario(sig, 8)),
        # sixteen models: the scan's loops over up to 16 models
        "sixteen_models": (sixteen, W.fc_scenario(sixteen, 9)),
    }


CASES = _cases()


def _near_options(prob, fc, f):
    tau = np.repeat(np.asarray(fc["tau"], np.float64), prob["n_options"])
    return np.abs(f - tau) <= NEAR * np.maximum(np.abs(tau), np.abs(f)) + 1e-7


def _fhat_condition(prob, fc):
    """Per option row: the condition scale of the raw throughput output under the
    observed state, sum of |weight| x |input| propagated along the layers
    (a1 = |W1||z| + |b1|, a2 = |W2| a1 + |b2|, c = |W3[0]| a_last + |b3[0]|): an
    fp32 evaluation in any order errs by a small multiple of 2^-24 of it."""
    n = np.asarray(prob["n_options"])
    d, h1, h2 = int(prob["d_local"]), int(prob["hidden1"]), int(prob["hidden2"])
    din, per = d + 4, W.param_count(d, h1, h2)
    N = n.size
    s_a = np.asarray(prob["agg_scale"] if prob.get("agg_scale") is not None else W.default_agg_scale(N),
                     np.float64)
    zobs = np.abs(np.asarray(fc["obs"], np.float64) * s_a)
    x = np.abs(np.asarray(prob["local_feats"], np.float64).reshape(-1, d))
    off = np.concatenate([[0], np.cumsum(n)])
    out = np.empty(int(off[-1]))
    for i in range(N):
        w = np.abs(np.asarray(prob["weights"], np.float64)[i * per:(i + 1) * per])
        o = 0
        W1 = w[o:o + h1 * din].reshape(h1, din); o += h1 * din
        b1 = w[o:o + h1]; o += h1
        z = np.concatenate([x[off[i]:off[i + 1]], np.broadcast_to(zobs, (int(n[i]), 4))], axis=1)
        a = z @ W1.T + b1
        if h2:
            W2 = w[o:o + h2 * h1].reshape(h2, h1); o += h2 * h1
            b2 = w[o:o + h2]; o += h2
            a = a @ W2.T + b2
        hl = h2 or h1
        W3 = w[o:o + 2 * hl].reshape(2, hl); o += 2 * hl
        out[off[i]:off[i + 1]] = a @ W3[0] + w[o]
    return out


@pytest.mark.parametrize("name", list(CASES))
def test_fc_table_matches_oracle(mf, oracle_mod, name):
    """Tolerances follow the arithmetic: the raw throughput errs by at most 1e-5 of
    its condition scale c; f = (fhat - f_min) / span by that over the span (plus its
    own rounding); the utility term by its slope in f, omega Q + 2 beta max(0, tau +
    delta - f), times f's error (plus rounding).  Floors within f's error of tau are
    near-threshold."""
    prob, fc = CASES[name]
    o = oracle_mod.Oracle(prob)
    rf, rff, rok, ru = o.fc_local(fc)
    with mf.Context(prob) as ctx:
        ctx.fc_set(fc)
        fhat, f, u, ok = ctx.fc_table()
    n = prob["n_options"]
    span = np.asarray(fc["f_max"], np.float64) - np.asarray(fc["f_min"], np.float64)
    tol_fhat = RTOL * _fhat_condition(prob, fc)
    tol_f = tol_fhat / span + 1e-6 * np.abs(rff)
    tau = np.repeat(np.asarray(fc["tau"], np.float64), n)
    slope = np.repeat(np.asarray(fc["omega"], np.float64), n) * np.asarray(fc["quality"], np.float64) + \
        2 * float(fc["beta"]) * np.maximum(tau + float(fc["delta"]) - rff, 0.0)
    tol_u = slope * tol_f + 1e-6 * np.maximum(1.0, np.abs(ru))
    assert np.all(np.abs(fhat - rf) <= tol_fhat)
    assert np.all(np.abs(f - rff) <= tol_f)
    assert np.all(np.abs(u - ru) <= tol_u)
    near = _near_options(prob, fc, rff) | (np.abs(rff - tau) <= tol_f)
    assert np.array_equal(ok[~near], rok[~near])


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("k", [1, 8, 32, 100])  # (up to 64: per-warp lists; 100: one list per CTA)
def test_fc_search_matches_oracle(mf, oracle_mod, name, k):
    prob, fc = CASES[name]
    o = oracle_mod.Oracle(prob)
    ti, ts, cnt = o.fc_exhaustive(fc, k)
    _, rff, _, ru = o.fc_local(fc)
    with mf.Context(prob) as ctx:
        ctx.fc_set(fc)
        res = ctx.fc_search(k)
    # candidates touching a near-floor option or near the VRAM cap may differ
    near_opt = _near_options(prob, fc, rff)
    n = o.space_size()
    idx = np.arange(n, dtype=np.uint64)
    digits = np.stack(np.unravel_index(idx.astype(np.int64), tuple(prob["n_options"])), axis=1)
    off = np.concatenate([[0], np.cumsum(prob["n_options"])[:-1]])
    rows = digits + off
    vram = prob["demand"][rows, 1].astype(np.float64).sum(axis=1)
    cap = float(prob["vram_cap"])
    near = near_opt[rows].any(axis=1) | (np.abs(vram - cap) <= NEAR * cap)
    assert abs(res["count"] - cnt) <= int(near.sum())
    tol = RTOL * max(1.0, float(np.abs(ru).sum()))
    got_i = np.asarray(res["topk_idx"], np.uint64)
    got_s = np.asarray(res["topk_score"], np.float64)
    fin = np.isfinite(ts)
    assert np.array_equal(np.isfinite(got_s), fin) or near.any()
    if fin.any():
        Jb, fb = o.fc_score_digits(fc, o.decode(int(got_i[0])))
        assert fb and abs(Jb - ts[0]) <= tol
        np.testing.assert_allclose(got_s[fin], ts[fin], rtol=0, atol=tol)


@pytest.mark.parametrize("name", ["tiny", "paper_vram_binds"])
def test_vram_feasible_list_matches_oracle(mf, oracle_mod, name):
    prob, _ = CASES[name]
    o = oracle_mod.Oracle(prob)
    c, lst = o.vram_feasible()
    with mf.Context(prob) as ctx:
        gc, gl = ctx.vram_feasible()
        assert gc == c and 0 < c < o.space_size()
        assert np.array_equal(gl.cpu().numpy().astype(np.uint64), lst)
        # a sub-range with a capacity below the count: counted in full, written in part
        lo, hi = o.space_size() // 7, o.space_size() - o.space_size() // 9
        c2, l2 = o.vram_feasible(lo, hi, cap=100)
        gc2, gl2 = ctx.vram_feasible(lo, hi, cap=100)
        assert gc2 == c2 and np.array_equal(gl2.cpu().numpy().astype(np.uint64), l2)


@pytest.mark.parametrize("which,seed,chunk", [("large", 3, 1 << 26), ("stress", 5, 1 << 30)])
def test_fc_full_size_separable_closed_form(mf, oracle_mod, which, seed, chunk):
    """At full size (24^6 and 16^8 candidates) the VRAM cap of 180 GB never binds, so
    the feasible count is the product of the per-model floor-feasible option counts
    and the best configuration takes each model's best feasible option (from the
    oracle's per-option table).  Chunks of 2^26 and 2^30 give the scan's threads short
    and long slices."""
    prob = W.large(precision="fp32") if which == "large" else W.stress(precision="fp32")
    fc = W.fc_scenario(prob, seed)
    o = oracle_mod.Oracle(prob)
    _, rff, rok, ru = o.fc_local(fc)
    assert not _near_options(prob, fc, rff).any()
    off = np.concatenate([[0], np.cumsum(prob["n_options"])])
    count, best, Jbest = 1, [], 0.0
    for i in range(len(prob["n_options"])):
        ui = np.where(rok[off[i]:off[i + 1]], ru[off[i]:off[i + 1]], -np.inf)
        count *= int(rok[off[i]:off[i + 1]].sum())
        best.append(int(np.argmax(ui)))
        Jbest += float(np.max(ui))
    with mf.Context(prob) as ctx:
        ctx.fc_set(fc)
        res = ctx.fc_search(16, chunk=chunk)
    assert res["count"] == count
    assert list(o.decode(res["best_idx"])) == best
    assert abs(res["best_score"] - Jbest) <= RTOL * max(1.0, float(np.abs(ru).sum()))


def test_fc_errors(mf):
    prob, fc = CASES["tiny"]
    with mf.Context(prob) as ctx:
        with pytest.raises(mf.MFError) as e:
            ctx.fc_search(4)
        assert e.value.status == mf.MF_EINVAL
        bad = dict(fc, f_max=np.asarray(fc["f_min"]).copy())
        with pytest.raises(mf.MFError) as e:
            ctx.fc_set(bad)
        assert e.value.status == mf.MF_EINVAL and "f_max" in str(e.value)


# ---------------------------------------------------------------------------
# The paper's GA on the fixed-context landscape
# ---------------------------------------------------------------------------

def _integer_fc(prob, seed):
    """Utility inputs that keep every term an integer on an integer landscape:
    f = fhat (f_min 0, f_max 1), Q and omega small integers, alpha = 1 with integer
    reload costs, beta = 0; floors integers."""
    fc = W.fc_scenario(prob, seed)
    rows = int(prob["n_options"].sum())
    n = int(prob["n_options"].size)
    rs = np.random.default_rng(seed)
    return dict(fc, f_min=np.zeros(rows, np.float32), f_max=np.ones(rows, np.float32),
                quality=rs.integers(1, 3, rows).astype(np.float32), omega=rs.integers(1, 3, n).astype(np.float32),
                reload_cost=rs.integers(1, 20, n).astype(np.float32), alpha=1.0, beta=0.0, delta=0.0,
                tau=rs.integers(-150, 0, n).astype(np.float32))


@pytest.mark.parametrize("opts,params", [
    ([12, 9, 9, 9, 9], dict(W.PAPER_GA_PARAMS)),
    ([12, 9, 9, 9, 9], dict(W.PAPER_GA_PARAMS, elitism=0, gens=12)),
    ([16] * 4, dict(W.PAPER_GA_PARAMS, pop=1024, gens=20, tournament=4, crossover_p=1.0, mutation_p=0.05)),
    ([5] * 8, dict(W.PAPER_GA_PARAMS, pop=37, repair=0)),
    ([200], dict(W.PAPER_GA_PARAMS, pop=2, gens=1)),
])
def test_paper_ga_reproduces_the_oracle_exactly(mf, oracle_mod, opts, params):
    """On an integer landscape every fitness is an exact integer, so the GPU run
    must equal the oracle's run: same decision, same fitness."""
    prob = W.integer_landscape(opts, 5, 5.0 * len(opts) + 5.0)
    fc = _integer_fc(prob, 7)
    o = oracle_mod.Oracle(prob)
    _, _, cnt = o.fc_exhaustive(fc, 1)
    assert 0 < cnt < o.space_size()
    with mf.Context(prob) as ctx:
        ctx.fc_set(fc)
        for seed in (1000, 1001, 2 ** 40 + 9):
            J, g = ctx.fc_ga_run(params, seed)
            Jo, go = o.fc_ga_run(fc, params, seed)
            assert list(g) == list(go) and J == Jo, (seed, g, go, J, Jo)


@pytest.mark.parametrize("case", ["floor_unmet", "vram_short", "vram_exact"])
def test_paper_ga_with_no_or_one_tier_of_feasible_configurations(mf, oracle_mod, case):
    """The GA kernel skips repairs when no configuration can be feasible (its repair draws
    have their own stream, so the run is the same as drawing every attempt in vain).
    floor_unmet: model 0 has no option at its floor; vram_short: every floor can be met
    but the smallest VRAM demands exceed the cap by 1; vram_exact: they equal the cap
    (feasible, the bound being inclusive).  Each run equals the oracle's bit for bit."""
    opts = [12, 9, 9, 9, 9]
    prob = W.integer_landscape(opts, 5, 5.0 * len(opts) + 5.0)
    fc = _integer_fc(prob, 7)
    if case == "floor_unmet":
        tau = np.asarray(fc["tau"], np.float32).copy()
        tau[0] = 1e6
        fc = dict(fc, tau=tau)
    else:
        _, _, rok, _ = oracle_mod.Oracle(prob).fc_local(fc)
        off = np.concatenate([[0], np.cumsum(prob["n_options"])])
        vram = np.asarray(prob["demand"], np.float64)[:, 1]
        need = sum(float(vram[off[i]:off[i + 1]][rok[off[i]:off[i + 1]]].min()) for i in range(len(opts)))
        prob = dict(prob, vram_cap=np.float32(need - 1.0 if case == "vram_short" else need))
    o = oracle_mod.Oracle(prob)
    _, _, cnt = o.fc_exhaustive(fc, 1)
    assert (cnt == 0) == (case != "vram_exact")
    params = dict(W.PAPER_GA_PARAMS, gens=12)
    with mf.Context(prob) as ctx:
        ctx.fc_set(fc)
        for seed in (1000, 2 ** 40 + 9):
            J, g = ctx.fc_ga_run(params, seed)
            Jo, go = o.fc_ga_run(fc, params, seed)
            assert list(g) == list(go) and (J == Jo or (np.isinf(J) and np.isinf(Jo))), (seed, g, go, J, Jo)


def test_paper_ga_decisions_on_the_paper_landscape(mf, oracle_mod):
    """The synthetic N = 5 landscape: every decision's oracle score equals its reported
    fitness and is within 0.5 % of the exhaustive optimum."""
    prob = W.paper_scale()
    o = oracle_mod.Oracle(prob)
    with mf.Context(prob) as ctx:
        for sc in W.GA_SCENARIO_SEEDS[:4]:
            fc = W.fc_scenario(prob, sc)
            _, ts, cnt = o.fc_exhaustive(fc, 1)
            if cnt == 0:
                continue
            ctx.fc_set(fc)
            for seed in (1000, 1001):
                J, g = ctx.fc_ga_run(W.PAPER_GA_PARAMS, seed)
                Jo, feas = o.fc_score_digits(fc, g)
                assert feas and abs(J - Jo) <= 1e-5 * max(1.0, abs(Jo))
                assert Jo >= ts[0] - 0.005 * abs(ts[0])


@pytest.mark.parametrize("chunk", [1 << 22, 1 << 30])
def test_fc_search_warp_lists_equal_cta_list(mf, chunk):
    """The scan keeps per-warp lists for k <= 64 and one list per CTA above: on the
    large space (24^6) the first 64 entries of a top-128 search (CTA list) equal a
    top-64 search (warp lists), and the counts agree."""
    prob = W.large(precision="fp32")
    fc = W.fc_scenario(prob, 3)
    with mf.Context(prob) as ctx:
        ctx.fc_set(fc)
        a = ctx.fc_search(64, chunk=chunk)
        b = ctx.fc_search(128, chunk=chunk)
    assert a["count"] == b["count"]
    np.testing.assert_array_equal(np.asarray(a["topk_idx"]), np.asarray(b["topk_idx"])[:64])
    np.testing.assert_array_equal(np.asarray(a["topk_score"]), np.asarray(b["topk_score"])[:64])
