"""GPU parity of the bf16 tensor-core path (tcgen05) against the CPU oracle.

Per-candidate scores within 2e-2 relative, feasibility exact away from the
bf16 band of the thresholds; exhaustive results are re-scored in fp32, so the
reported top-k meets the fp32 bar and the chosen configuration is optimal within
1e-5 relative."""
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


def _problems():
    paper = W.paper_scale(precision="bf16")
    tight = W.paper_scale(precision="bf16")
    W.set_scenario(tight, 17, W.TIGHT_SLA)
    # the stress per-model shape (d_L 16 -> K1 = 32, 128-wide layers, soft latency)
    # on three models, so all weights fit shared memory
    stress3 = W.make_problem([16] * 3, 16, 128, 128, 4, 180.0, objective="soft_lat",
                             soft_penalty=0.1, precision="bf16", sla_range=(-0.2, 0.3))
    # odd d_L (padded), one hidden layer, sigmoid outputs, binding VRAM cap
    odd = W.make_problem([7, 9, 6], 7, 32, 0, 12, 30.0, out_act="sigmoid", precision="bf16",
                         sla_range=(0.4, 0.9))
    # paper's 64-32 predictor shape, eight models (16 D3 columns)
    p6432 = W.make_problem([4] * 8, 8, 64, 32, 13, 100.0, precision="bf16", sla_range=W.TIGHT_SLA)
    # five 20->128->128->2 models: 240 KB of bf16 weights, staged in two passes (3 + 2 models)
    multipass = W.make_problem([3, 4, 2, 3, 2], 16, 128, 128, 5, 180.0, precision="bf16",
                               sla_range=(0.2, 0.8))
    return {"paper": paper, "tight": tight, "stress3": stress3, "odd": odd, "p6432": p6432,
            "multipass": multipass}


PROBLEMS = _problems()


def _score(ctx, idx_np):
    import torch
    idx = torch.from_numpy(idx_np.astype(np.int64)).cuda()
    s, f, p = ctx.score_batch(idx, with_pred=True)
    torch.cuda.synchronize()
    return s.cpu().numpy(), f.cpu().numpy(), p.cpu().numpy()


@pytest.mark.parametrize("name", list(PROBLEMS))
def test_tc_score_batch_matches_oracle(mf, oracle_mod, name):
    prob = PROBLEMS[name]
    o = oracle_mod.Oracle(prob)
    n = o.space_size()
    rs = np.random.default_rng(1)
    idx = np.arange(n, dtype=np.uint64) if n <= 40000 else rs.integers(0, n, 40000).astype(np.uint64)
    with mf.Context(prob) as ctx:
        assert ctx.precision == "bf16"
        s, f, p = _score(ctx, idx)
        assert ctx.check_status() == mf.MF_OK
    r = o.score_list(idx, with_pred=True)
    near = check_scores(prob, s, f, *r, prec="bf16", got_pred=p, pred_scale=o.pred_scale(idx))
    assert near < 0.5 * idx.size


def test_tc_ragged_tail_and_single_candidate(mf, oracle_mod):
    prob = PROBLEMS["tight"]
    o = oracle_mod.Oracle(prob)
    with mf.Context(prob) as ctx:
        for n in (1, 127, 129, 1000, 128 * 4 * 152 + 77):
            idx = (np.arange(n, dtype=np.uint64) * 7919) % np.uint64(o.space_size())
            s, f, p = _score(ctx, idx)
            check_scores(prob, s, f, *o.score_list(idx, with_pred=True), prec="bf16", got_pred=p,
                         pred_scale=o.pred_scale(idx))


def test_tc_out_of_range_index(mf):
    import torch
    prob = PROBLEMS["paper"]
    with mf.Context(prob) as ctx:
        idx = torch.tensor([0, 78732, 5], dtype=torch.int64, device="cuda")
        s, f = ctx.score_batch(idx)
        assert ctx.check_status() == mf.MF_EDEVICE
        assert s.cpu().numpy()[1] == -np.inf and f.cpu().numpy()[1] == 0


@pytest.mark.parametrize("name", list(PROBLEMS))
@pytest.mark.parametrize("k", [1, 32])
def test_tc_exhaustive_matches_oracle(mf, oracle_mod, name, k):
    prob = PROBLEMS[name]
    o = oracle_mod.Oracle(prob)
    ti, ts, cnt = o.exhaustive(k)
    n = o.space_size()
    _, _, pr, ag = o.score_list(np.arange(n, dtype=np.uint64), with_pred=True)
    bound = int(near_threshold(prob, pr, ag, "bf16").sum())
    with mf.Context(prob) as ctx:
        res = ctx.search(k)
    check_search(o, prob, res, k, (ti, ts), cnt, near_count_bound=bound, prec="bf16")


@pytest.mark.parametrize("chunk", [1 << 12, 77777, 0])
def test_tc_chunk_invariance(mf, chunk):
    prob = PROBLEMS["tight"]
    with mf.Context(prob) as ctx:
        ref = ctx.search(32, chunk=1 << 20)
        got = ctx.search(32, chunk=chunk)
    assert got["count"] == ref["count"]
    assert np.array_equal(got["topk_idx"], ref["topk_idx"])


def test_tc_and_fp32_paths_agree_on_large_range(mf):
    """A 2^22-candidate range of the N=6 workload searched by both paths: the
    re-scored bf16 top-k equals the fp32 top-k (the bf16 path re-scores its shortlist
    with the CUDA-core fp32 kernels, so against precision fp32_simt)."""
    lo, hi = 24 ** 6 // 2, 24 ** 6 // 2 + (1 << 22)
    with mf.Context(W.large(precision="fp32"), precision="fp32_simt") as c32, \
            mf.Context(W.large(precision="bf16")) as c16:
        a = c32.search(32, lo=lo, hi=hi)
        b = c16.search(32, lo=lo, hi=hi)
    assert a["count"] == b["count"] == hi - lo
    np.testing.assert_array_equal(a["topk_idx"], b["topk_idx"])
    np.testing.assert_allclose(a["topk_score"], b["topk_score"], rtol=1e-5, atol=1e-6)
