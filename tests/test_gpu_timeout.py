"""The failure path of the bounded device waits, made to run on the GPU without a
fault or a hang: mf_debug_wait_test makes each waiting kernel first wait on a flag
that nothing sets, with a bound of a few polls.  The wait runs out, the kernel flags
the context's status and runs to its end (draining only its own MMAs and copies),
the call reports MF_ETIMEOUT, and the context gives correct results again once the
test wait is switched off."""
import numpy as np
import pytest

from paper_2609_02109_gb300 import workload as W

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


def test_scorer_wait_gives_up_and_the_context_recovers(mf):
    prob = W.paper_scale(precision="bf16")
    with mf.Context(prob, precision="bf16") as ref_ctx:
        ref = ref_ctx.search(8)
    with mf.Context(prob, precision="bf16") as ctx:
        ctx.debug_wait_test(2)
        with pytest.raises(mf.MFError) as e:
            ctx.search(8)
        assert e.value.status == mf.MF_ETIMEOUT
        ctx.debug_wait_test(0)
        got = ctx.search(8)
    assert got["count"] == ref["count"] and got["best_idx"] == ref["best_idx"]
    np.testing.assert_array_equal(got["topk_idx"], ref["topk_idx"])
    np.testing.assert_array_equal(got["topk_score"], ref["topk_score"])


def test_ga_wait_gives_up_and_the_context_recovers(mf, oracle_mod):
    prob = W.integer_landscape([12, 9, 9, 9, 9], 5, 30.0)
    g = dict(W.GA_PARAMS, gens=20)
    with mf.Context(prob) as ctx:
        ctx.debug_wait_test(3)
        with pytest.raises(mf.MFError) as e:
            ctx.ga_run(g, 1000)
        assert e.value.status == mf.MF_ETIMEOUT
        ctx.debug_wait_test(0)
        J, genome = ctx.ga_run(g, 1000)
    Jo, go = oracle_mod.Oracle(prob).ga_run(g, 1000)
    assert J == Jo and list(genome) == list(go)
