"""The multi-GPU path's host logic on CPU ranks (gloo, world size 2).

bench.py shards the questions across ranks (each rank a replica of the
corpus and its own batch; no data-path collective) and reports the maximum
of the ranks' times.  Here two gloo ranks draw their batches exactly as the
benchmark does and check that together they are the single-rank batch of
2 Q questions, split at a question boundary with rebased offsets, and that
the timing reduction returns the maximum."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import synth

SPEC = synth.WorkloadSpec("shard_test", 7, 5000, 64, "bf16", 6, (1, 9), 5, 8, "clustered", 16)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        corpus, scale, regions, offsets = bench.make_inputs(SPEC, rank, world, "cpu")
        t = bench.max_over_ranks(float(rank + 1) * 1.5, world)
        out[rank] = (synth.bf16_bits(corpus), synth.bf16_bits(regions), offsets.numpy(), t)
    finally:
        dist.destroy_process_group()


def test_two_ranks_partition_the_questions():
    world = 2
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    port = _free_port()
    mp.start_processes(_rank, args=(world, port, out), nprocs=world, start_method="spawn", join=True)
    # The single-rank draw of 2 Q questions.
    centres = synth.draw_centres(SPEC, SPEC.centres, SPEC.d)
    all_regions, all_offsets = synth.make_regions(SPEC, centres, "cpu", Q=SPEC.Q * world)
    all_bits = synth.bf16_bits(all_regions)
    r0 = 0
    for rank in range(world):
        c_bits, reg_bits, offs, t = out[rank]
        assert t == 3.0  # max over ranks of 1.5 and 3.0
        q0 = rank * SPEC.Q
        lo, hi = int(all_offsets[q0]), int(all_offsets[q0 + SPEC.Q])
        assert lo == r0
        assert offs[0] == 0 and offs[-1] == hi - lo and len(offs) == SPEC.Q + 1
        assert (offs == (all_offsets[q0:q0 + SPEC.Q + 1].numpy() - lo)).all()
        assert (reg_bits == all_bits[lo:hi]).all()
        r0 = hi
    assert r0 == all_bits.shape[0]
    # Every rank holds the same corpus replica.
    assert (out[0][0] == out[1][0]).all()
