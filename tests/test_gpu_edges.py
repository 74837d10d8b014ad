"""Edge shapes of the scorer on both GPU paths against the oracle: a single model, models
with a single option, the maximum of 16 models (a 32-column layer-3 accumulator on the
tensor-core path), 255 options per model and a joint space beyond 2^32 (64-bit digit
decoding), including its last index."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

from _parity import check_scores, check_search, near_threshold

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def mf():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_02109_gb300 import build
    build.build()
    from paper_2609_02109_gb300 import mf as mod
    return mod


def _shapes():
    return {
        # one model: the aggregate is the model's own demand; the VRAM cap binds
        "one_model": ([37], 8, 64, 64, 31, 12.0, (0.3, 1.0)),
        # models with a single option (a digit that never changes)
        "single_options": ([5, 1, 6, 1], 8, 32, 0, 32, 62.0, (0.0, 0.6)),
        # sixteen models: n3 = 32 on the tensor-core path
        "sixteen_models": ([2] * 16, 8, 32, 32, 33, 180.0, (0.4, 1.2)),
        # 255 options per model, |Lambda| = 255^5 > 2^32
        "beyond_2_32": ([255] * 5, 8, 64, 64, 34, 60.0, (0.3, 1.5)),
    }


SHAPES = _shapes()
PRECISIONS = ["fp32", "bf16"]


def _prob(name, prec):
    ks, dl, h1, h2, seed, cap, sla = SHAPES[name]
    return W.make_problem(ks, dl, h1, h2, seed, cap, precision=prec, sla_range=sla)


def _score(ctx, idx_np):
    import torch
    idx = torch.from_numpy(idx_np.astype(np.int64)).cuda()
    s, f, p = ctx.score_batch(idx, with_pred=True)
    torch.cuda.synchronize()
    return s.cpu().numpy(), f.cpu().numpy(), p.cpu().numpy()


def _indices(n):
    if n <= 40000:
        return np.arange(n, dtype=np.uint64)
    rs = np.random.default_rng(5)
    body = rs.integers(0, n, 20000, dtype=np.uint64)
    ends = np.array([0, 1, n // 2, n - 2, n - 1], dtype=np.uint64)
    return np.concatenate([ends, body])


@pytest.mark.parametrize("prec", PRECISIONS)
@pytest.mark.parametrize("name", list(SHAPES))
def test_edge_score_batch_matches_oracle(mf, oracle_mod, name, prec):
    prob = _prob(name, prec)
    o = oracle_mod.Oracle(prob)
    idx = _indices(o.space_size())
    with mf.Context(prob) as ctx:
        assert ctx.precision == prec
        s, f, p = _score(ctx, idx)
        assert ctx.check_status() == mf.MF_OK
    r = o.score_list(idx, with_pred=True)
    kw = dict(got_pred=p)
    if prec == "bf16":
        kw["pred_scale"] = o.pred_scale(idx)
    near = check_scores(prob, s, f, *r, prec=prec, **kw)
    assert near < 0.5 * idx.size
    assert 0 < int(np.asarray(f).astype(bool).sum()) < idx.size  # both masks are exercised


@pytest.mark.parametrize("prec", PRECISIONS)
@pytest.mark.parametrize("name", ["one_model", "single_options", "sixteen_models"])
def test_edge_exhaustive_matches_oracle(mf, oracle_mod, name, prec):
    prob = _prob(name, prec)
    o = oracle_mod.Oracle(prob)
    k = 32
    ti, ts, cnt = o.exhaustive(k)
    n = o.space_size()
    _, _, pr, ag = o.score_list(np.arange(n, dtype=np.uint64), with_pred=True)
    bound = int(near_threshold(prob, pr, ag, prec).sum())
    with mf.Context(prob) as ctx:
        res = ctx.search(k)
    check_search(o, prob, res, k, (ti, ts), cnt, near_count_bound=bound, prec=prec)


@pytest.mark.parametrize("prec", PRECISIONS)
def test_range_at_the_top_of_a_space_beyond_2_32(mf, oracle_mod, prec):
    """The last 2^18 + 3 indices of 255^5: digits decoded in 64 bits, the final index
    included, a ragged tail."""
    prob = _prob("beyond_2_32", prec)
    o = oracle_mod.Oracle(prob)
    n = o.space_size()
    assert n > 2 ** 32
    lo, hi = n - (1 << 18) - 3, n
    k = 16
    ti, ts, cnt = o.exhaustive(k, lo=lo, hi=hi)
    _, _, pr, ag = o.score_list(np.arange(lo, hi, dtype=np.uint64), with_pred=True)
    bound = int(near_threshold(prob, pr, ag, prec).sum())
    with mf.Context(prob) as ctx:
        res = ctx.search(k, lo=lo, hi=hi)
    check_search(o, prob, res, k, (ti, ts), cnt, near_count_bound=bound, prec=prec)
    assert 0 < cnt < hi - lo
