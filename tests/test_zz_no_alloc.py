"""mf_search_exhaustive_noalloc: the exhaustive search for callers that cannot
allocate device memory (for example a serving process whose memory pool already
holds the GPU's memory, or a control loop that must not pay cudaMalloc's implicit
synchronisation).  It keeps all of its device memory in one fixed array inside the
library.  Its results must equal those of the regular entry point,
mf_search_exhaustive, on every call, including consecutive calls that reuse the
array left behind by the previous one.  It runs the CUDA-core fp32 kernels, so it is
compared with contexts of precision "fp32_simt".

This file is named to be collected last, so a run that stops at the first failure
has already run every other test."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

pytestmark = pytest.mark.gpu

RTOL = 1e-5  # the fp32 path's score tolerance


@pytest.fixture(scope="module")
def mf():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_02109_gb300 import build
    build.build()
    from paper_2609_02109_gb300 import mf as mod
    return mod


def _tight():
    p = W.paper_scale()
    return W.set_scenario(p, 17, W.TIGHT_SLA)


def _same(got, ref):
    assert got["count"] == ref["count"]
    assert got["best_idx"] == ref["best_idx"]
    np.testing.assert_array_equal(got["topk_idx"], ref["topk_idx"])
    fin = np.isfinite(ref["topk_score"])
    assert np.array_equal(fin, np.isfinite(got["topk_score"]))
    np.testing.assert_allclose(got["topk_score"][fin], ref["topk_score"][fin], rtol=RTOL, atol=0)


@pytest.mark.parametrize("k", [1, 32, 64])
def test_noalloc_equals_regular_search_on_consecutive_calls(mf, k):
    problems = [W.tiny(), _tight(), W.paper_scale()]
    refs = []
    for prob in problems:  # (the same CUDA-core fp32 kernels)
        with mf.Context(prob, precision="fp32_simt") as ctx:
            refs.append(ctx.search(k))
    # two calls in a row on each problem, then the problems in a different order:
    # each call must clear what the previous call left in the shared array
    for prob, ref in zip(problems, refs):
        for _ in range(2):
            _same(mf.search_exhaustive_noalloc(prob, k), ref)
    for j in (2, 0, 1):
        _same(mf.search_exhaustive_noalloc(problems[j], k, chunk=1 << 12), refs[j])


def test_noalloc_rejects_sizes_beyond_its_limits(mf):
    with pytest.raises(mf.MFError) as e:
        mf.search_exhaustive_noalloc(W.tiny(), 65)
    assert e.value.status == mf.MF_EINVAL and "64" in str(e.value)
    # six 20->256->256->2 predictors: 6 x 287 KB of fp32 weights > the 1 MiB limit
    big = W.make_problem([4] * 6, 16, 256, 256, 1, 100.0)
    assert 6 * 4 * W.param_count(16, 256, 256) > (1 << 20)
    with pytest.raises(mf.MFError) as e:
        mf.search_exhaustive_noalloc(big, 8)
    assert e.value.status == mf.MF_EINVAL and "MF_NOALLOC_MAX_WEIGHT_BYTES" in str(e.value)


def test_noalloc_allocates_nothing_after_the_first_call(mf):
    """The first call on a device reserves the array (the runtime loads the module
    that holds it); later calls must leave the device's free memory exactly as it
    was.  For contrast, creating a context and searching with it does allocate."""
    import torch
    prob = W.paper_scale()
    mf.search_exhaustive_noalloc(prob, 8)  # the first call on this device
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for k in (1, 8, 64):
        mf.search_exhaustive_noalloc(prob, k)
        mf.search_exhaustive_noalloc(W.tiny(), k, chunk=1 << 10)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    with mf.Context(prob) as ctx:
        ctx.search(8)
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] < free0


def test_noalloc_matches_the_oracle(mf, oracle_mod):
    """The same result as the CPU oracle's exhaustive search (fp64 on the same fp32
    inputs), under the search contract of the other parity tests: the count within
    the number of candidates near a threshold, every reported entry feasible and
    scored within the fp32 tolerance, indices exact where scores are well separated,
    on a problem whose SLA mask binds."""
    from _parity import check_search, near_threshold
    prob = _tight()
    o = oracle_mod.Oracle(prob)
    ti, ts, cnt = o.exhaustive(32)
    _, _, pr, ag = o.score_list(np.arange(o.space_size(), dtype=np.uint64), with_pred=True)
    bound = int(near_threshold(prob, pr, ag).sum())
    assert 0 < cnt < o.space_size()
    res = mf.search_exhaustive_noalloc(prob, 32)
    check_search(o, prob, res, 32, (ti, ts), cnt, near_count_bound=bound)
