"""The multi-GPU split and exchange of the exhaustive search, on CPU ranks (gloo).

Each rank searches its index range with the oracle (standing in for its GPU) and
the ranks exchange and merge through paper_2609_02109_gb300.shard; the merged result
must equal the oracle's single-range search of the whole space."""
import os
import socket

import numpy as np
import pytest

from paper_2609_02109_gb300 import shard
from paper_2609_02109_gb300 import workload as W


def test_shard_ranges_cover_the_space():
    for total, world in [(78732, 2), (216, 4), (5, 8), (0, 3), (2 ** 32, 7)]:
        spans = [shard.shard_range(total, r, world) for r in range(world)]
        assert spans[0][0] == 0 and spans[-1][1] == total
        for (a, b), (c, d) in zip(spans, spans[1:]):
            assert b == c and b >= a
        sizes = [b - a for a, b in spans]
        assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        shard.shard_range(10, 2, 2)


def test_merge_orders_by_score_then_index_and_pads():
    a = dict(topk_idx=np.array([5, 9, shard.EMPTY], np.uint64), topk_score=np.array([2.0, 1.0, -np.inf], np.float32),
             count=2)
    b = dict(topk_idx=np.array([3, 7, 8], np.uint64), topk_score=np.array([2.0, 1.0, 0.5], np.float32), count=3)
    m = shard.merge_results([a, b], 4)
    assert list(m["topk_idx"]) == [3, 5, 7, 9] and m["count"] == 5 and m["best_idx"] == 3
    m = shard.merge_results([a, dict(topk_idx=np.full(3, shard.EMPTY, np.uint64),
                                     topk_score=np.full(3, -np.inf, np.float32), count=0)], 4)
    assert list(m["topk_idx"]) == [5, 9, shard.EMPTY, shard.EMPTY] and m["count"] == 2


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, k, name, out_dir):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from oracle import oracle
    prob = {"tight": W.set_scenario(W.paper_scale(), 17, W.TIGHT_SLA), "tiny": W.tiny()}[name]
    o = oracle.Oracle(prob)
    lo, hi = shard.shard_range(o.space_size(), rank, world)
    ti, ts, cnt = o.exhaustive(k, lo=lo, hi=hi)
    local = dict(topk_idx=np.asarray(ti, np.uint64), topk_score=np.asarray(ts, np.float32), count=cnt)
    merged = shard.gather_merge(local, k)
    np.savez(os.path.join(out_dir, f"r{rank}.npz"), idx=merged["topk_idx"], score=merged["topk_score"],
             count=merged["count"])
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world,k,name", [(2, 32, "tight"), (3, 8, "tiny"), (2, 300, "tiny")])
def test_gloo_ranks_merge_to_the_single_range_result(oracle_mod, tmp_path, world, k, name):
    import torch.multiprocessing as mp
    mp.start_processes(_rank_main, args=(world, _free_port(), k, name, str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    prob = {"tight": W.set_scenario(W.paper_scale(), 17, W.TIGHT_SLA), "tiny": W.tiny()}[name]
    ti, ts, cnt = oracle_mod.Oracle(prob).exhaustive(k)
    for r in range(world):
        got = np.load(tmp_path / f"r{r}.npz")
        assert int(got["count"]) == cnt
        assert np.array_equal(got["idx"], np.asarray(ti, np.uint64))
        assert np.array_equal(got["score"], np.asarray(ts, np.float32))


class _OracleContext:
    """The two members of the binding's Context that search_sharded uses (space_size,
    search over an index range), served by the oracle: a rank's GPU on the CPU."""

    def __init__(self, prob):
        from oracle import oracle
        self.o = oracle.Oracle(prob)
        self.space_size = self.o.space_size()

    def search(self, k, lo=0, hi=None, chunk=0):
        ti, ts, cnt = self.o.exhaustive(k, lo=lo, hi=hi)
        return dict(best_idx=int(ti[0]), best_score=float(ts[0]), count=cnt,
                    topk_idx=np.asarray(ti, np.uint64), topk_score=np.asarray(ts, np.float32))


def _sharded_main(rank, world, port, k, out_dir):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    prob = W.set_scenario(W.paper_scale(), 17, W.TIGHT_SLA)
    merged = shard.search_sharded(_OracleContext(prob), k)
    np.savez(os.path.join(out_dir, f"s{rank}.npz"), idx=merged["topk_idx"], score=merged["topk_score"],
             count=merged["count"], best=merged["best_idx"])
    dist.barrier()
    dist.destroy_process_group()


def test_search_sharded_end_to_end_on_gloo_ranks(oracle_mod, tmp_path):
    """The multi-GPU step of the benchmark (shard.search_sharded: this rank's range,
    then the all-gather and merge) on two CPU ranks equals the single search."""
    import torch.multiprocessing as mp
    world, k = 2, 32
    mp.start_processes(_sharded_main, args=(world, _free_port(), k, str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    prob = W.set_scenario(W.paper_scale(), 17, W.TIGHT_SLA)
    ti, ts, cnt = oracle_mod.Oracle(prob).exhaustive(k)
    for r in range(world):
        got = np.load(tmp_path / f"s{r}.npz")
        assert int(got["count"]) == cnt and int(got["best"]) == int(ti[0])
        assert np.array_equal(got["idx"], np.asarray(ti, np.uint64))
        assert np.array_equal(got["score"], np.asarray(ts, np.float32))
