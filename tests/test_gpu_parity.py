"""GPU parity of the exact fp32 path (C ABI -> CUDA kernels) against the CPU
oracle on the same seeded inputs."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

from _parity import check_scores, check_search

pytestmark = pytest.mark.gpu

EMPTY = 2 ** 64 - 1


@pytest.fixture(scope="module")
def mf():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_02109_gb300 import build
    build.build()
    from paper_2609_02109_gb300 import mf as mod
    return mod


def _torch():
    import torch
    return torch


def _score_all(ctx, idx_np, with_pred=True):
    torch = _torch()
    idx = torch.from_numpy(idx_np.astype(np.int64)).cuda()
    out = ctx.score_batch(idx, with_pred=with_pred)
    torch.cuda.synchronize()
    return [t.cpu().numpy() for t in out]


def _problems():
    tight = W.paper_scale()
    W.set_scenario(tight, 17, W.TIGHT_SLA)
    sig = W.random_small(21, n_models=4, max_options=8, h2=32, vram_cap=40.0, out_act="sigmoid",
                         sla_range=(0.4, 0.9))
    soft = W.make_problem([3] * 8, 16, 128, 128, 4, 180.0, objective="soft_lat", soft_penalty=0.1,
                          sla_range=(-0.2, 0.3))
    odd = W.make_problem([5, 7, 3], 3, 20, 10, 8, 30.0, sla_range=W.TIGHT_SLA)
    return {"hand": W.hand_example(), "tiny": W.tiny(), "paper": W.paper_scale(), "tight": tight,
            "sigmoid": sig, "soft8": soft, "odd_shape": odd}


PROBLEMS = _problems()


@pytest.mark.parametrize("name", list(PROBLEMS))
def test_score_batch_all_candidates(mf, oracle_mod, name):
    prob = PROBLEMS[name]
    o = oracle_mod.Oracle(prob)
    n = o.space_size()
    idx = np.arange(n, dtype=np.uint64)
    if n > 50000:
        idx = np.random.default_rng(0).permutation(n)[:50000].astype(np.uint64)
    with mf.Context(prob) as ctx:
        s, f, p = _score_all(ctx, idx)
        assert ctx.check_status() == mf.MF_OK
    rs, rf, rp, ra = o.score_list(idx, with_pred=True)
    check_scores(prob, s, f, rs, rf, rp, ra, got_pred=p)


@pytest.mark.parametrize("name", list(PROBLEMS))
@pytest.mark.parametrize("k", [1, 8, 32])
def test_exhaustive_matches_oracle(mf, oracle_mod, name, k):
    prob = PROBLEMS[name]
    o = oracle_mod.Oracle(prob)
    ti, ts, cnt = o.exhaustive(k)
    with mf.Context(prob) as ctx:
        res = ctx.search(k)
    n_idx = np.arange(o.space_size(), dtype=np.uint64)
    _, _, pr, ag = o.score_list(n_idx, with_pred=True) if o.space_size() <= 100000 else (None,) * 4
    from _parity import near_threshold
    bound = int(near_threshold(prob, pr, ag).sum()) if pr is not None else 0
    check_search(o, prob, res, k, (ti, ts), cnt, near_count_bound=bound)


def test_hand_example_exact_values(mf):
    with mf.Context(W.hand_example()) as ctx:
        res = ctx.search(4)
    assert res["count"] == 2 and res["best_idx"] == 1
    assert list(res["topk_idx"][:2]) == [1, 0]
    np.testing.assert_allclose(res["topk_score"][:2], [0.85, 0.8], rtol=1e-6)
    assert list(res["topk_idx"][2:]) == [EMPTY, EMPTY]
    assert np.all(res["topk_score"][2:] == -np.inf)


@pytest.mark.parametrize("chunk", [1 << 10, 1 << 14, 77777, 0])
def test_chunk_size_invariance(mf, chunk):
    with mf.Context(W.paper_scale()) as ctx:
        ref = ctx.search(32, chunk=1 << 20)
        got = ctx.search(32, chunk=chunk)
    assert got["count"] == ref["count"]
    assert np.array_equal(got["topk_idx"], ref["topk_idx"])
    assert np.array_equal(got["topk_score"], ref["topk_score"])


@pytest.mark.parametrize("lo,hi", [(0, 0), (5, 6), (1000, 1000 + 4099), (78732 - 513, 78732)])
def test_range_search_matches_oracle(mf, oracle_mod, lo, hi):
    prob = PROBLEMS["tight"]
    o = oracle_mod.Oracle(prob)
    ti, ts, cnt = o.exhaustive(16, lo=lo, hi=hi)
    with mf.Context(prob) as ctx:
        res = ctx.search(16, lo=lo, hi=hi)
    check_search(o, prob, res, 16, (ti, ts), cnt)
    assert all(lo <= int(i) < hi for i in res["topk_idx"] if int(i) != EMPTY)


def test_large_k_and_no_feasible(mf):
    prob = W.tiny()
    with mf.Context(prob) as ctx:
        res = ctx.search(1024)
        assert np.sum(res["topk_idx"] != np.uint64(EMPTY)) == res["count"]
    prob = W.tiny()
    prob["vram_cap"] = 0.5
    with mf.Context(prob) as ctx:
        res = ctx.search(8)
    assert res["count"] == 0 and res["best_idx"] == EMPTY and res["best_score"] == -np.inf


def test_order_invariance_of_score_batch(mf):
    prob = PROBLEMS["tight"]
    rs = np.random.default_rng(5)
    idx = rs.integers(0, 78732, size=30000).astype(np.uint64)
    perm = rs.permutation(idx.size)
    with mf.Context(prob) as ctx:
        s1, f1, _ = _score_all(ctx, idx)
        s2, f2, _ = _score_all(ctx, idx[perm])
    assert np.array_equal(s1[perm], s2) and np.array_equal(f1[perm], f2)


def test_out_of_range_index_raises_device_status(mf):
    torch = _torch()
    with mf.Context(W.tiny()) as ctx:
        idx = torch.tensor([0, 5, 216, 3], dtype=torch.int64, device="cuda")
        s, f = ctx.score_batch(idx)
        assert ctx.check_status() == mf.MF_EDEVICE
        assert ctx.check_status() == mf.MF_OK  # cleared
        s = s.cpu().numpy()
        assert s[2] == -np.inf and np.isfinite(s[0]) or s[0] == -np.inf
        pop = torch.tensor([[0, 0], [12, 1]], dtype=torch.int32, device="cuda")
        fit = ctx.ga_generation(pop)
        assert ctx.check_status() == mf.MF_EDEVICE
        assert fit.cpu().numpy()[1] == -np.inf


def test_set_objective_changes_scores(mf, oracle_mod):
    prob = W.paper_scale()
    with mf.Context(prob) as ctx:
        W.set_scenario(prob, 123, (-0.1, 0.8))
        ctx.set_objective(prob["sla"], prob["obj_w"])
        res = ctx.search(8)
    o = oracle_mod.Oracle(prob)
    ti, ts, cnt = o.exhaustive(8)
    check_search(o, prob, res, 8, (ti, ts), cnt, near_count_bound=50)


# ---------------------------------------------------------------------------
# GA operators: bit-exact against the oracle on the same inputs.
# ---------------------------------------------------------------------------

def test_ga_init_bit_exact(mf, oracle_mod):
    prob = W.paper_scale()
    o = oracle_mod.Oracle(prob)
    g = dict(W.GA_PARAMS)
    with mf.Context(prob) as ctx:
        for seed in (1000, 1001, 2 ** 63 + 5):
            pop = ctx.ga_init(g, seed).cpu().numpy()
            assert np.array_equal(pop, o.ga_init(g, seed))


@pytest.mark.parametrize("elitism", [0, 1])
@pytest.mark.parametrize("gen", [0, 1, 57])
def test_ga_step_bit_exact(mf, oracle_mod, elitism, gen):
    torch = _torch()
    prob = W.ga_scenario(101)
    W.set_scenario(prob, 101, (-0.2, 0.4))
    o = oracle_mod.Oracle(prob)
    g = dict(W.GA_PARAMS, elitism=elitism)
    pop = o.ga_init(g, 7)
    s, _ = o.score_list(np.zeros(1, dtype=np.uint64))  # warm the oracle
    fit64 = np.array([o.score_digits(row)[0] for row in pop])
    fit32 = fit64.astype(np.float32)          # what a float32 fitness batch carries
    fit32[10:20] = fit32[5]                   # ties exercise the lowest-slot rule
    ref = o.ga_step(g, 7, gen, pop, fit32.astype(np.float64))
    with mf.Context(prob) as ctx:
        nxt = ctx.ga_step(g, 7, gen, torch.from_numpy(pop).cuda(), torch.from_numpy(fit32).cuda())
        got = nxt.cpu().numpy()
    assert np.array_equal(got, ref)


def test_ga_generation_matches_oracle(mf, oracle_mod):
    torch = _torch()
    prob = W.ga_scenario(102)
    W.set_scenario(prob, 102, (-0.2, 0.4))
    o = oracle_mod.Oracle(prob)
    g = dict(W.GA_PARAMS)
    pop = o.ga_init(g, 3)
    idx = np.ravel_multi_index(tuple(pop.T), prob["n_options"]).astype(np.uint64)
    rs, rf, rp, ra = o.score_list(idx, with_pred=True)
    with mf.Context(prob) as ctx:
        fit = ctx.ga_generation(torch.from_numpy(pop).cuda()).cpu().numpy()
    check_scores(prob, fit, np.isfinite(fit), rs, rf, rp, ra)


def test_ga_run_finds_tiny_optimum(mf, oracle_mod):
    prob = W.tiny()
    o = oracle_mod.Oracle(prob)
    ti, ts, _ = o.exhaustive(1)
    with mf.Context(prob) as ctx:
        J, genome = ctx.ga_run(dict(W.GA_PARAMS, pop=64, gens=30), 1000)
    assert list(genome) == list(o.decode(int(ti[0])))
    assert abs(J - ts[0]) <= 1e-5 * abs(ts[0])


def test_ga_run_reports_oracle_score_of_its_genome(mf, oracle_mod):
    prob = W.ga_scenario(100)
    o = oracle_mod.Oracle(prob)
    with mf.Context(prob) as ctx:
        for seed in (1000, 1001):
            J, genome = ctx.ga_run(W.GA_PARAMS, seed)
            Jo, f, pred, _ = o.score_digits(genome)
            assert f and abs(J - Jo) <= 1e-5 * max(abs(Jo), float(np.abs(pred[:, 0]) @ prob["obj_w"]))
            assert 0 <= genome.min() and all(genome < prob["n_options"])


@pytest.mark.parametrize("world", [2, 3, 7])
def test_index_range_shards_merge_to_the_full_search(mf, world):
    """The multi-GPU split run rank by rank on one GPU: every shard's range search,
    merged by the exchange step's merge, equals the single search of the space."""
    from paper_2609_02109_gb300 import shard
    prob = PROBLEMS["tight"]
    with mf.Context(prob) as ctx:
        full = ctx.search(32)
        parts = [ctx.search(32, *shard.shard_range(ctx.space_size, r, world)) for r in range(world)]
    m = shard.merge_results(parts, 32)
    assert m["count"] == full["count"] and m["best_idx"] == full["best_idx"]
    assert np.array_equal(m["topk_idx"], full["topk_idx"])
    assert np.array_equal(m["topk_score"], full["topk_score"])
