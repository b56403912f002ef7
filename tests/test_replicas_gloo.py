"""Two replicas of the pruned prefill as gloo ranks on the CPU: the host side
of a run on several GPUs, which has no collective on the data path.

Each rank draws its own token shard and runs the float64 oracle on it,
standing in for its GPU's forward. It meets the other rank at the barrier
and takes the slowest rank's step time; the job throughput counts both
ranks' tokens. The checks:
- the shards are distinct and fixed by the rank;
- every rank reports the same (slowest) step time;
- the two ranks' results equal one process's run over the joined batch.
Sequences never read one another (Sec. 3 prunes within a sequence), so the
replicas need no exchange."""

import os
import socket
import time

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

from oracle import zsaa_oracle as O
from paper_2509_01190_gb300 import inputs as I
from paper_2509_01190_gb300 import replicas as R
from tests.helpers import oracle_cfg

WORLD, B, L, ACCEL = 2, 2, 48, 2.0


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, port, out_dir):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=WORLD)
    try:
        shape = I.TINY_F32
        w = I.weights_to_numpy(I.make_weights(shape))
        tokens = I.make_tokens(B, L, shape.vocab, seed=R.rank_token_seed(I.TOKEN_SEED, rank))
        R.barrier(dist)
        t0 = time.perf_counter()
        res = O.forward(oracle_cfg(shape), w, tokens, accel=ACCEL)
        ms_local = 1e3 * (time.perf_counter() - t0)
        ms = R.max_over_ranks(ms_local, dist)
        all_ms = [None] * WORLD
        dist.all_gather_object(all_ms, ms_local)
        R.barrier(dist)
        np.savez(os.path.join(out_dir, f"rank{rank}.npz"), tokens=tokens, logits=res["logits"],
                 kept=res["kept_pos"], ms=ms, all_ms=np.array(all_ms),
                 tps=R.job_tokens_per_s(WORLD, B, L, ms))
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas(tmp_path):
    mp.spawn(_rank_main, args=(_free_port(), str(tmp_path)), nprocs=WORLD, join=True)
    r = [np.load(tmp_path / f"rank{k}.npz") for k in range(WORLD)]
    shape = I.TINY_F32
    # distinct shards, each fixed by its rank
    assert not np.array_equal(r[0]["tokens"], r[1]["tokens"])
    for k in range(WORLD):
        np.testing.assert_array_equal(r[k]["tokens"], I.make_tokens(B, L, shape.vocab, seed=I.TOKEN_SEED + k))
    # one step time for the job: the slowest rank's, seen by every rank
    slowest = float(np.max(r[0]["all_ms"]))
    np.testing.assert_array_equal(r[0]["all_ms"], r[1]["all_ms"])
    for k in range(WORLD):
        assert float(r[k]["ms"]) == slowest
        assert float(r[k]["tps"]) == pytest.approx(WORLD * B * L / (slowest / 1e3), rel=1e-12)
    # no exchange needed: one process over the joined batch gives the same results
    w = I.weights_to_numpy(I.make_weights(shape))
    both = O.forward(oracle_cfg(shape), w, np.concatenate([r[0]["tokens"], r[1]["tokens"]]), accel=ACCEL)
    np.testing.assert_array_equal(both["kept_pos"], np.concatenate([r[0]["kept"], r[1]["kept"]]))
    np.testing.assert_allclose(both["logits"], np.concatenate([r[0]["logits"], r[1]["logits"]]),
                               rtol=1e-12, atol=1e-12)
