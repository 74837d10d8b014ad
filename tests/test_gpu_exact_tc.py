"""The exact fp32 tensor-core variant: precision "fp32" on the d_L 8, 12 -> 64 -> 64 -> 2
predictor shape (Eq. 6) scores on the tensor cores with every operand split into two
tf32 parts (hi.hi + hi.lo + lo.hi, fp32 accumulation).  It must meet the fp32 contract
(1e-5 relative, feasibility exact away from thresholds) against the oracle and agree
with the CUDA-core fp32 path ("fp32_simt") to the same tolerance.  N = 5 and 6 run in
two weight passes (three models per pass); N = 2 in one."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W
from _parity import check_scores, check_search, near_threshold, score_scale, RTOL

pytestmark = pytest.mark.gpu

PATH_SIMT, PATH_BF16, PATH_EXACT = 0, 1, 2


@pytest.fixture(scope="module")
def mf():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_02109_gb300 import build
    build.build()
    from paper_2609_02109_gb300 import mf as mod
    return mod


def _score_all(ctx, idx_np):
    import torch
    idx = torch.from_numpy(idx_np.astype(np.int64)).cuda()
    out = ctx.score_batch(idx, with_pred=True)
    torch.cuda.synchronize()
    return [t.cpu().numpy() for t in out]


def _cases():
    tight = W.set_scenario(W.paper_scale(), 17, W.TIGHT_SLA)
    two = W.make_problem([23, 19], 8, 64, 64, 11, 30.0, sla_range=W.TIGHT_SLA)
    soft = W.make_problem([5, 6, 4, 7, 3, 5], 8, 64, 64, 12, 60.0, objective="soft_lat", soft_penalty=0.1,
                          sla_range=(0.1, 0.6))
    return {"paper": W.paper_scale(), "tight": tight, "two_models": two, "soft6": soft}


CASES = _cases()


def test_scoring_paths(mf):
    paper = W.paper_scale()
    with mf.Context(paper) as c:
        assert c.stats()["scoring_path"] == PATH_EXACT
    with mf.Context(paper, precision="fp32_simt") as c:
        assert c.stats()["scoring_path"] == PATH_SIMT
    with mf.Context(paper, precision="bf16") as c:
        assert c.stats()["scoring_path"] == PATH_BF16
    with mf.Context(W.tiny()) as c:  # 12 -> 32 -> 2: the CUDA cores
        assert c.stats()["scoring_path"] == PATH_SIMT


@pytest.mark.parametrize("name", list(CASES))
def test_exact_score_batch_matches_oracle_and_simt(mf, oracle_mod, name):
    prob = CASES[name]
    o = oracle_mod.Oracle(prob)
    n = o.space_size()
    idx = np.arange(n, dtype=np.uint64)
    if n > 40000:
        idx = np.random.default_rng(1).permutation(n)[:40000].astype(np.uint64)
    with mf.Context(prob) as ctx:
        assert ctx.stats()["scoring_path"] == PATH_EXACT
        s, f, p = _score_all(ctx, idx)
        assert ctx.check_status() == mf.MF_OK
    with mf.Context(prob, precision="fp32_simt") as ctx:
        s2, f2, p2 = _score_all(ctx, idx)
    rs, rf, rp, ra = o.score_list(idx, with_pred=True)
    check_scores(prob, s, f, rs, rf, rp, ra, got_pred=p)
    # the two fp32 paths: the same feasibility away from thresholds, scores within 2e-5
    near = near_threshold(prob, rp, ra)
    assert np.array_equal(f.astype(bool)[~near], f2.astype(bool)[~near])
    both = f.astype(bool) & f2.astype(bool)
    scale = np.maximum(score_scale(prob, rs, rp), 1e-30)
    assert np.all(np.abs(s[both].astype(np.float64) - s2[both]) <= 2 * RTOL["fp32"] * scale[both])


@pytest.mark.parametrize("name", ["paper", "tight", "soft6"])
@pytest.mark.parametrize("k", [1, 32])
def test_exact_search_matches_oracle(mf, oracle_mod, name, k):
    prob = CASES[name]
    o = oracle_mod.Oracle(prob)
    ti, ts, cnt = o.exhaustive(k)
    _, _, pr, ag = o.score_list(np.arange(o.space_size(), dtype=np.uint64), with_pred=True)
    with mf.Context(prob) as ctx:
        res = ctx.search(k)
        assert ctx.check_status() == mf.MF_OK
    check_search(o, prob, res, k, (ti, ts), cnt, near_count_bound=int(near_threshold(prob, pr, ag).sum()))


def test_exact_and_simt_searches_agree_on_the_large_space(mf, oracle_mod):
    """24^6 (six models, two weight passes), a range of 2^22 candidates in chunks of
    2^20: the same count (the latency mask does not bind here) and top-32 scores within
    the fp32 tolerance of the terms' scale (the oracle's rescoring of the entries), the
    same indices where the scores are well separated."""
    prob = W.large(precision="fp32")
    lo = 123_456_789
    with mf.Context(prob) as ctx:
        assert ctx.stats()["scoring_path"] == PATH_EXACT
        a = ctx.search(32, lo=lo, hi=lo + (1 << 22), chunk=1 << 20)
    with mf.Context(prob, precision="fp32_simt") as ctx:
        b = ctx.search(32, lo=lo, hi=lo + (1 << 22), chunk=1 << 20)
    assert a["count"] == b["count"] == 1 << 22
    o = oracle_mod.Oracle(prob)
    s_o, f_o, pred_o, _ = o.score_list(np.asarray(b["topk_idx"], np.uint64), with_pred=True)
    assert f_o.all()
    scale = np.maximum(score_scale(prob, s_o, pred_o), 1e-30)
    sa, sb = a["topk_score"].astype(np.float64), b["topk_score"].astype(np.float64)
    assert np.all(np.abs(sa - sb) <= 2 * RTOL["fp32"] * scale)
    assert np.all(np.abs(sb - s_o) <= RTOL["fp32"] * scale)
    gaps = np.abs(np.diff(s_o))
    sep = (np.r_[gaps, np.inf] > 4 * RTOL["fp32"] * scale) & (np.r_[np.inf, gaps] > 4 * RTOL["fp32"] * scale)
    assert np.array_equal(np.asarray(a["topk_idx"])[sep], np.asarray(b["topk_idx"])[sep])


def test_exact_search_with_the_longest_lists(mf, oracle_mod):
    """k = 1024 (the API's maximum; the exact variant's lists then share shared memory
    with a three-model weight pass, or the search runs on the CUDA cores where they do
    not fit): the count and the list of fp32_simt, scores within the fp32 tolerance."""
    prob = W.paper_scale()
    with mf.Context(prob) as ctx:
        a = ctx.search(1024)
    with mf.Context(prob, precision="fp32_simt") as ctx:
        b = ctx.search(1024)
    assert a["count"] == b["count"]
    o = oracle_mod.Oracle(prob)
    fin = np.isfinite(b["topk_score"])
    s_o, _, pred_o, _ = o.score_list(np.asarray(b["topk_idx"], np.uint64)[fin], with_pred=True)
    scale = np.maximum(score_scale(prob, s_o, pred_o), 1e-30)
    assert np.array_equal(np.isfinite(a["topk_score"]), fin)
    assert np.all(np.abs(a["topk_score"][fin].astype(np.float64) - b["topk_score"][fin]) <= 2 * RTOL["fp32"] * scale)
    gaps = np.abs(np.diff(s_o))
    sep = (np.r_[gaps, np.inf] > 4 * RTOL["fp32"] * scale) & (np.r_[np.inf, gaps] > 4 * RTOL["fp32"] * scale)
    assert np.array_equal(np.asarray(a["topk_idx"])[fin][sep], np.asarray(b["topk_idx"])[fin][sep])
