"""Bounded waits: a tensor-core launch whose every wait may give up at once
reports SKIP_ETIMEOUT through skip_sync_status, frees its resources, and the
same handle then works normally.  No fault or hang is involved: the kernel's
waits are bounded by the option, and after giving up each role waits (up to
a second) for its copies and MMAs in flight before the CTA exits."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_25422_gb300 as skip
import synth
from tests import checker

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("mma", [1, 2])
def test_wait_timeout_reports_and_recovers(mma):
    dev = torch.device("cuda")
    N, d, R, k = 60000, 256, 300, 12
    ct = synth.random_bf16(N, d, seed=91)
    rt = synth.random_bf16(R, d, seed=92)
    c = skip.skip_corpus_load(ct.to(dev))
    try:
        c.set_option(skip.SKIP_OPT_PATH, skip.SKIP_PATH_TENSOR)
        c.set_option(skip.SKIP_OPT_MMA, mma)
        c.set_option(skip.SKIP_OPT_WAIT_TIMEOUT_NS, 0)
        reg = rt.to(dev)
        skip.skip_retrieve_regions(c, reg, k)
        assert skip.skip_sync_status(c) == skip.SKIP_ETIMEOUT
        # The error word was cleared by the report; the context is usable.
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        c.set_option(skip.SKIP_OPT_WAIT_TIMEOUT_NS, 2_000_000_000)
        rid, rsc = skip.skip_retrieve_regions(c, reg, k)
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        rid, rsc = rid.cpu().numpy(), rsc.cpu().numpy()
    finally:
        c.free()
    cn, rn = synth.bf16_bits(ct), synth.bf16_bits(rt)
    ids_ext, sc_ext = oracle.region_topk(cn, rn[:40], k + 32)
    for r, t in enumerate(checker.region_truths(ids_ext, sc_ext, k)):
        _, probs = checker.check_region(rid[r], rsc[r], t)
        assert not probs, (r, probs)
