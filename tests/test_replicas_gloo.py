"""The N > 1 path: independent replicas, one per rank, on CPU over gloo.

Each rank drafts and verifies its own batch with the oracle (the data path
has no collective, so what a rank computes must not depend on the others),
then the launcher logic combines the per-rank timings. Run as two spawned
processes with world size 2.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
import synth
from paper_2607_07409_gb300 import replicas


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _draft(w):
    d = synth.make_inputs(w, device="cpu")
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    res = oracle.draft_block(oracle.make_head(w.head, W), d["long"], oracle.log_prior(d["counts"]), w.alpha,
                             w.beta)
    acc, bonus, _ = oracle.verify_greedy(res.tokens, d["target"])
    return res.tokens, np.asarray(acc), np.asarray(bonus)


def _worker(rank, world, port, out_dir):
    os.environ.update(WORLD_SIZE=str(world), RANK=str(rank), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    info = replicas.rank_info()
    dist.init_process_group("gloo", rank=info.rank, world_size=info.world)
    try:
        base = synth.with_sizes(synth.stress(synth.WORKLOADS["tiny"]), B=3)
        w = synth.with_sizes(base, seed=replicas.replica_seed(base.seed, info.rank))
        replicas.barrier()
        tok, acc, bonus = _draft(w)
        # each rank reports a different time; the job time is the slowest rank's
        ms = 10.0 * (info.rank + 1)
        ms_max = replicas.max_over_ranks(ms)
        gathered = [None] * info.world
        dist.all_gather_object(gathered, (tok.tolist(), acc.tolist(), bonus.tolist()))
        value = replicas.job_throughput([w.B * w.n] * info.world, ms_max)
        replicas.barrier()
        if info.rank == 0:
            torch.save({"gathered": gathered, "ms_max": ms_max, "value": value, "B": w.B, "n": w.n},
                       os.path.join(out_dir, "result.pt"))
    finally:
        dist.destroy_process_group()


def test_two_replicas_match_independent_runs(tmp_path):
    world = 2
    mp.start_processes(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, start_method="spawn",
                       join=True)
    r = torch.load(os.path.join(tmp_path, "result.pt"))
    assert r["ms_max"] == 20.0
    assert r["value"] == pytest.approx(world * r["B"] * r["n"] / 0.020)
    base = synth.with_sizes(synth.stress(synth.WORKLOADS["tiny"]), B=3)
    outs = []
    for rank in range(world):
        tok, acc, bonus = _draft(synth.with_sizes(base, seed=replicas.replica_seed(base.seed, rank)))
        g_tok, g_acc, g_bonus = r["gathered"][rank]
        np.testing.assert_array_equal(np.asarray(g_tok), tok)
        np.testing.assert_array_equal(np.asarray(g_acc), acc)
        np.testing.assert_array_equal(np.asarray(g_bonus), bonus)
        outs.append(tok)
    # the two replicas drafted different requests
    assert not np.array_equal(outs[0], outs[1])


@pytest.mark.parametrize("total,world", [(64, 1), (64, 2), (64, 8), (7, 3), (2, 4), (0, 2)])
def test_request_ranges_partition_the_batch(total, world):
    seen = []
    sizes = []
    for rank in range(world):
        a, b = replicas.request_range(total, world, rank)
        assert 0 <= a <= b <= total
        seen.extend(range(a, b))
        sizes.append(b - a)
    assert seen == list(range(total))
    assert max(sizes) - min(sizes) <= 1


def test_single_process_helpers():
    assert replicas.max_over_ranks(3.5) == 3.5
    assert replicas.replica_seed(3, 0) == 3
    assert len({replicas.replica_seed(3, r) for r in range(8)}) == 8
    with pytest.raises(ValueError):
        replicas.job_throughput([1.0], 0.0)
