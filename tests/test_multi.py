"""The several-GPU path's host logic on CPU: two gloo ranks, each with a
stand-in context whose pbs_batch is the CPU oracle, shard a batch, take the
maximum of their times and gather the outputs on rank 0."""

import os
import socket

import numpy as np
import pytest

from paper_2609_16915_gb300 import multi


def test_shard_range_partitions():
    for total in [0, 1, 7, 16, 4096, 4097]:
        for world in [1, 2, 3, 8]:
            spans = [multi.shard_range(total, world, r) for r in range(world)]
            assert spans[0][0] == 0
            for (s0, c0), (s1, _) in zip(spans, spans[1:]):
                assert s0 + c0 == s1
            assert sum(c for _, c in spans) == total
            assert max(c for _, c in spans) - min(c for _, c in spans) <= 1
    with pytest.raises(ValueError):
        multi.shard_range(10, 2, 2)


class _OracleCtx:
    """Stand-in for a Context: same call, computed by the CPU oracle."""

    def __init__(self, p, keys):
        self.p, self.keys = p, keys

    def pbs_batch(self, lwe, lut, out):
        import oracle as O
        out[:] = O.pbs_batch(self.p, self.keys.bsk, self.keys.ksk, lwe, lut, threads=2)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, result_path):
    import torch.distributed as dist

    import oracle as O
    import workload as W
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p), threads=1)
    lwe = W.uniform_ciphertexts(p, 7, sub=5)        # 7 rows: uneven slices
    lut = W.lut_torus(p)
    got = multi.pbs_batch_sharded(_OracleCtx(p, keys), lwe, lut, dist)
    slowest = multi.max_over_ranks(1.0 + rank, dist)
    if rank == 0:
        want = O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut, threads=2)
        np.save(result_path, np.array([np.array_equal(got, want), slowest == float(world)]))
    else:
        assert got is None
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_and_gather(tmp_path):
    import torch.multiprocessing as mp
    result = str(tmp_path / "result.npy")
    mp.start_processes(_rank_main, args=(2, _free_port(), result), nprocs=2, start_method="spawn", join=True)
    ok_gather, ok_max = np.load(result)
    assert ok_gather and ok_max
