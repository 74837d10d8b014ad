"""The Eq. 3 utility on the coupled aggregate (mf_set_utility) through the fp32 and
bf16 scorers, the exhaustive search and the GA, against the oracle's util_* functions.

Tolerances follow the arithmetic: a predicted throughput fhat_i errs by 1e-5 (fp32)
or 2e-2 (bf16) of its condition scale c_i (the oracle's sum of |terms| of the output
dot product); the utility term is a function of f_i = (fhat_i - f_min) / span with
slope omega_i Q_i + 2 beta max(0, tau_i + delta - f_i), so J errs by at most
sum_i slope_i * rtol * c_i / span_i (plus rounding of the sum).  Floors within that
error of tau_i and VRAM sums within 1e-4 of the cap are near-threshold."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

pytestmark = pytest.mark.gpu

RTOL = {"fp32": 1e-5, "bf16": 2e-2}


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
    tight["vram_cap"] = 55.0
    sig = W.random_small(21, n_models=4, max_options=8, h2=32, vram_cap=40.0, out_act="sigmoid")
    return {"paper": (W.paper_scale(), 3), "paper_vram_binds": (tight, 6), "sigmoid": (sig, 8)}


CASES = _cases()


def _bounds(o, prob, fc, idx, prec):
    """Per candidate: oracle J, feasibility, tolerance of J, near-threshold flag."""
    s, f, pred, agg = o.util_score_list(fc, idx, with_pred=True)
    cond = o.pred_scale(idx)[..., 0]
    n = prob["n_options"]
    off = np.concatenate([[0], np.cumsum(n)[:-1]])
    digits = np.stack(np.unravel_index(idx.astype(np.int64), tuple(n)), axis=1)
    rows = digits + off
    span = (np.asarray(fc["f_max"], np.float64) - np.asarray(fc["f_min"], np.float64))[rows]
    fmin = np.asarray(fc["f_min"], np.float64)[rows]
    fn = (pred[..., 0] - fmin) / span
    tau = np.asarray(fc["tau"], np.float64)[None, :]
    margin = np.maximum(tau + float(np.float32(fc["delta"])) - fn, 0.0)
    slope = np.asarray(fc["omega"], np.float64)[None, :] * np.asarray(fc["quality"], np.float64)[rows] + \
        2 * float(np.float32(fc["beta"])) * margin
    df = RTOL[prec] * cond / span
    tol = (slope * df).sum(axis=1) + 1e-6 * np.maximum(1.0, np.abs(np.where(np.isfinite(s), s, 0.0)))
    near = (np.abs(fn - tau) <= df + 1e-4 * np.maximum(np.abs(tau), np.abs(fn))).any(axis=1)
    near |= np.abs(agg[:, 1] - float(prob["vram_cap"])) <= 1e-4 * float(prob["vram_cap"])
    return s, f, tol, near


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
@pytest.mark.parametrize("name", list(CASES))
def test_util_score_batch(mf, oracle_mod, name, prec):
    import torch
    base, seed = CASES[name]
    prob = dict(base, precision=prec)
    fc = W.fc_scenario(prob, seed)
    o = oracle_mod.Oracle(prob)
    idx = np.random.default_rng(3).integers(0, o.space_size(), 20000).astype(np.uint64)
    s, f, tol, near = _bounds(o, prob, fc, idx, prec)
    with mf.Context(prob) as ctx:
        ctx.set_utility(fc)
        gs, gf = ctx.score_batch(torch.from_numpy(idx.astype(np.int64)).cuda())
        gs, gf = gs.cpu().numpy().astype(np.float64), gf.cpu().numpy().astype(bool)
    assert 0 < f.sum() < f.size
    bad = (gf != f) & ~near
    assert not bad.any(), np.where(bad)[0][:5]
    both = gf & f
    assert np.all(np.abs(gs[both] - s[both]) <= tol[both])


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
@pytest.mark.parametrize("name", list(CASES))
def test_util_search(mf, oracle_mod, name, prec):
    base, seed = CASES[name]
    prob = dict(base, precision=prec)
    fc = W.fc_scenario(prob, seed)
    o = oracle_mod.Oracle(prob)
    ti, ts, cnt = o.util_exhaustive(fc, 16)
    all_idx = np.arange(o.space_size(), dtype=np.uint64)
    _, _, tol, near = _bounds(o, prob, fc, all_idx, prec)
    with mf.Context(prob) as ctx:
        ctx.set_utility(fc)
        res = ctx.search(16)
        ctx.set_utility(None)
        plain = ctx.search(16)
    assert abs(res["count"] - cnt) <= int(near.sum())
    # the reported top-k are fp32 (bf16: re-scored) utility values of their indices
    gi = np.asarray(res["topk_idx"], np.uint64)
    s_at, f_at = o.util_score_list(fc, gi)
    fin = np.isfinite(np.asarray(res["topk_score"], np.float64))
    assert np.all(f_at[fin])
    _, _, tol_at, _ = _bounds(o, prob, fc, gi, "fp32")
    assert np.all(np.abs(np.asarray(res["topk_score"], np.float64)[fin] - s_at[fin]) <= tol_at[fin])
    # the choice is within tolerance of the optimum
    assert s_at[0] >= ts[0] - tol[int(ti[0])] - tol_at[0]
    # back to the problem's own objective
    ref_i, ref_s, ref_c = o.exhaustive(16)
    assert plain["count"] == ref_c or prec == "bf16"


def test_util_ga(mf, oracle_mod):
    prob = W.ga_scenario(103)
    fc = W.fc_scenario(prob, 3)
    o = oracle_mod.Oracle(prob)
    ti, ts, _ = o.util_exhaustive(fc, 1)
    with mf.Context(prob) as ctx:
        ctx.set_utility(fc)
        for seed in (1000, 1001):
            J, genome = ctx.ga_run(W.GA_PARAMS, seed)
            assert ctx.stats()["kernel_launches_last"] == 1
            Jo, feas, _ = o.util_score_digits(fc, genome)
            assert feas and abs(J - Jo) <= 1e-5 * max(1.0, abs(Jo))
            assert Jo >= ts[0] - 0.05 * abs(ts[0])  # a GA decision close to the optimum
