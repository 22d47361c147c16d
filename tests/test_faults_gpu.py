"""Debugging aids that stand in for tools closed on the GPU pool.

* Host-side fault injection: SKIP_FAULT_INJECT=alloc[:kind] makes the
  library's device allocations fail as on an exhausted device.  The corpus
  load and the workspace growth must return SKIP_ENOMEM, leave no handle
  behind, and leave an existing handle usable: its next call (with the
  variable cleared) allocates again and gives the oracle's lists.
* Canaries: with SKIP_OPT_CANARY the library puts guard bytes after its
  workspace, staging and gate buffers and skip_sync_status checks them; the
  test also puts guard words after out_ids / out_scores (and the per-region
  outputs) and checks them after the small cases and a full-size one.
None of this faults or stalls the GPU: the failures are made on the host.
"""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2607_25422_gb300 as skip
import synth
from tests import checker
from tests.test_parity_gpu import assert_parity, oracle_truth, ragged_offsets

pytestmark = pytest.mark.gpu

GUARD = 64  # guard elements after each output


@pytest.fixture
def inject():
    """Sets SKIP_FAULT_INJECT for the test and always clears it."""
    def set_(value):
        if value is None:
            os.environ.pop("SKIP_FAULT_INJECT", None)
        else:
            os.environ["SKIP_FAULT_INJECT"] = value
    yield set_
    os.environ.pop("SKIP_FAULT_INJECT", None)


def test_corpus_load_reports_enomem(inject):
    dev = torch.device("cuda")
    ct = synth.random_bf16(3000, 64, seed=1).to(dev)
    for value in ("alloc", "alloc:corpus"):
        inject(value)
        with pytest.raises(skip.SkipError) as e:
            skip.skip_corpus_load(ct)
        assert e.value.status == skip.SKIP_ENOMEM
    inject("alloc:workspace")  # another kind: the load itself succeeds
    c = skip.skip_corpus_load(ct)
    c.free()


@pytest.mark.parametrize("path", ["tensor", "warp", "latency"])
def test_workspace_growth_failure_leaves_handle_usable(inject, path):
    dev = torch.device("cuda")
    N, d, R, Q, k, K = 9000, 128, 20, 4, 12, 25
    ct = synth.random_bf16(N, d, seed=2)
    rt = synth.random_bf16(R, d, seed=3)
    offsets = ragged_offsets(Q, R, seed=4)
    c = skip.skip_corpus_load(ct.to(dev))
    try:
        c.set_option(skip.SKIP_OPT_PATH, {"tensor": skip.SKIP_PATH_TENSOR, "warp": skip.SKIP_PATH_WARP,
                                          "latency": skip.SKIP_PATH_LATENCY}[path])
        reg, off = rt.to(dev), torch.as_tensor(offsets).to(dev)
        inject("alloc:workspace")
        with pytest.raises(skip.SkipError) as e:
            skip.skip_retrieve(c, reg, off, k, K)
        assert e.value.status == skip.SKIP_ENOMEM
        with pytest.raises(skip.SkipError) as e:
            skip.skip_retrieve_host(c, rt.pin_memory(), torch.as_tensor(offsets), k, K)
        assert e.value.status == skip.SKIP_ENOMEM
        inject(None)
        rid, rsc = skip.skip_retrieve_regions(c, reg, k)
        oid, osc = skip.skip_retrieve(c, reg, off, k, K)
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        plan = skip.skip_last_plan(c)
        gpu = tuple(x.cpu().numpy() for x in (rid, rsc, oid, osc)) + (plan,)
    finally:
        c.free()
    cn, rn = synth.bf16_bits(ct), synth.bf16_bits(rt)
    assert_parity(cn, rn, offsets, k, K, gpu, oracle_truth(cn, rn, offsets, k, K))


def _guarded(shape, dtype, dev, fill):
    n = int(np.prod(shape))
    buf = torch.full((n + GUARD,), fill, dtype=dtype, device=dev)
    return buf, buf[:n].view(*shape)


CANARY_CASES = [
    # N, d, R, Q, k, K, path, mma, bound
    (30000, 256, 300, 20, 16, 40, skip.SKIP_PATH_TENSOR, 2, 1),
    (70000, 768, 512, 32, 20, 50, skip.SKIP_PATH_TENSOR, 2, 2),
    (12000, 512, 130, 9, 100, 100, skip.SKIP_PATH_TENSOR, 1, 1),
    (20000, 256, 30, 4, 10, 30, skip.SKIP_PATH_LATENCY, 0, 0),
    (5000, 128, 7, 3, 13, 20, skip.SKIP_PATH_WARP, 0, 0),
]


@pytest.mark.parametrize("case", CANARY_CASES, ids=lambda c: "N%d_R%d_k%d_path%d" % (c[0], c[2], c[4], c[6]))
def test_canaries_small(case):
    N, d, R, Q, k, K, path, mma, bound = case
    dev = torch.device("cuda")
    ct = synth.random_bf16(N, d, seed=N + 1)
    rt = synth.random_bf16(R, d, seed=R + 2)
    offsets = ragged_offsets(Q, R, seed=N + R)
    c = skip.skip_corpus_load(ct.to(dev))
    try:
        c.set_option(skip.SKIP_OPT_CANARY, 1)
        c.set_option(skip.SKIP_OPT_PATH, path)
        c.set_option(skip.SKIP_OPT_MMA, mma)
        c.set_option(skip.SKIP_OPT_BOUND, bound)
        reg, off = rt.to(dev), torch.as_tensor(offsets).to(dev)
        rib, rid = _guarded((R, k), torch.int64, dev, 0x5A5A5A5A)
        rsb, rsc = _guarded((R, k), torch.float32, dev, 12345.0)
        oib, oid = _guarded((Q, K), torch.int64, dev, 0x5A5A5A5A)
        osb, osc = _guarded((Q, K), torch.float32, dev, 12345.0)
        skip.skip_retrieve_regions(c, reg, k, rid, rsc)
        skip.skip_retrieve(c, reg, off, k, K, oid, osc)
        hi = torch.empty(Q * K + GUARD, dtype=torch.int64).fill_(0x5A5A5A5A).pin_memory()
        hs = torch.empty(Q * K + GUARD, dtype=torch.float32).fill_(12345.0).pin_memory()
        skip.skip_retrieve_host(c, rt.pin_memory(), torch.as_tensor(offsets), k, K, hi[:Q * K].view(Q, K),
                                hs[:Q * K].view(Q, K))
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        plan = skip.skip_last_plan(c)
        for b in (rib, oib, hi):
            assert torch.all(b[-GUARD:].cpu() == 0x5A5A5A5A)
        for b in (rsb, osb, hs):
            assert torch.all(b[-GUARD:].cpu() == 12345.0)
        np.testing.assert_array_equal(hi[:Q * K].view(Q, K).numpy(), oid.cpu().numpy())
        gpu = tuple(x.cpu().numpy() for x in (rid, rsc, oid, osc)) + (plan,)
        c.set_option(skip.SKIP_OPT_CANARY, 0)
    finally:
        c.free()
    cn, rn = synth.bf16_bits(ct), synth.bf16_bits(rt)
    assert_parity(cn, rn, offsets, k, K, gpu, oracle_truth(cn, rn, offsets, k, K))


def test_canaries_full_size_clustered_1m():
    """The 1M-row workload in the launch configuration the benchmark times,
    with guards: the library's guard bytes and the output guards intact."""
    spec = synth.WORKLOADS["clustered_1m"]
    dev = torch.device("cuda")
    corpus, _, centres = synth.make_corpus(spec, device=dev)
    regions, offsets = synth.make_regions(spec, centres, "cpu")
    R, Q, k, K = regions.shape[0], spec.Q, spec.k_region, spec.K
    c = skip.skip_corpus_load(corpus)
    del corpus
    try:
        c.set_option(skip.SKIP_OPT_CANARY, 1)
        reg, off = regions.to(dev), offsets.to(dev)
        oib, oid = _guarded((Q, K), torch.int64, dev, 0x5A5A5A5A)
        osb, osc = _guarded((Q, K), torch.float32, dev, 12345.0)
        for _ in range(3):
            skip.skip_retrieve(c, reg, off, k, K, oid, osc)
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        assert torch.all(oib[-GUARD:].cpu() == 0x5A5A5A5A)
        assert torch.all(osb[-GUARD:].cpu() == 12345.0)
        ids = oid.cpu().numpy()
        assert np.all(ids >= 0) and np.all(ids < spec.N)
    finally:
        c.free()
