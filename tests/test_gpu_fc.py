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
    return {
        "hand": (W.hand_example(), _hand_fc()),
        "tiny": (W.tiny(), W.fc_scenario(W.tiny(), 4)),
        "paper": (W.paper_scale(), W.fc_scenario(W.paper_scale(), 3)),
        "paper_vram_binds": (tight, W.fc_scenario(tight, 6)),
        "sigmoid": (sig, W.fc_scenario(sig, 8)),
    }


CASES = _cases()


def _near_options(prob, fc, f):
    tau = np.repeat(np.asarray(fc["tau"], np.float64), prob["n_options"])
    return np.abs(f - tau) <= NEAR * np.maximum(np.abs(tau), np.abs(f)) + 1e-7


@pytest.mark.parametrize("name", list(CASES))
def test_fc_table_matches_oracle(mf, oracle_mod, name):
    prob, fc = CASES[name]
    o = oracle_mod.Oracle(prob)
    rf, rff, rok, ru = o.fc_local(fc)
    with mf.Context(prob) as ctx:
        ctx.fc_set(fc)
        fhat, f, u, ok = ctx.fc_table()
    scale = np.maximum(np.abs(rf), 1.0)
    np.testing.assert_allclose(fhat, rf, rtol=0, atol=RTOL * 10)
    span = np.asarray(fc["f_max"], np.float64) - np.asarray(fc["f_min"], np.float64)
    np.testing.assert_allclose(f, rff, rtol=0, atol=RTOL * 10 * np.max(scale / span))
    np.testing.assert_allclose(u, ru, rtol=0, atol=RTOL * 100 * max(1.0, float(np.max(np.abs(ru)))))
    near = _near_options(prob, fc, rff)
    assert np.array_equal(ok[~near], rok[~near])


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("k", [1, 8, 32])
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


@pytest.mark.parametrize("which,seed", [("large", 3), ("stress", 5)])
def test_fc_full_size_separable_closed_form(mf, oracle_mod, which, seed):
    """At full size (24^6 and 16^8 candidates) the VRAM cap of 180 GB never binds, so
    the feasible count is the product of the per-model floor-feasible option counts
    and the best configuration takes each model's best feasible option (from the
    oracle's per-option table)."""
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
        res = ctx.fc_search(16, chunk=1 << 26)
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
