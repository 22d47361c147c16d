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


def test_gate_wait_timeout_reports_and_recovers():
    """The retrieval plus SKV gate with every wait allowed to give up at once
    (the gate's MLP waits for its flag, its TMA and MMA phases and its
    partner's half of the sums): SKIP_ETIMEOUT, then a normal call on the
    same handle whose gate matches the oracle on the call's own merged lists."""
    from tests.test_skv_gpu import check_gate
    dev = torch.device("cuda")
    N, d, Q, R_per, k, K = 20000, 128, 16, 4, 20, 50
    ct = synth.random_bf16(N, d, seed=93)
    rt = synth.random_bf16(Q * R_per, d, seed=94)
    offs = torch.arange(0, Q * R_per + 1, R_per, dtype=torch.int32)
    qbar = synth.random_bf16(Q, d, seed=95)
    vbar = synth.random_bf16(Q, d, seed=96)
    w1, b1, w2, b2 = synth.make_skv_mlp(d, 512, seed=97)
    t = lambda x: x.to(dev).contiguous()
    c = skip.skip_corpus_load(ct.to(dev))
    try:
        c.set_option(skip.SKIP_OPT_PATH, skip.SKIP_PATH_TENSOR)
        c.set_option(skip.SKIP_OPT_WAIT_TIMEOUT_NS, 0)
        args = (c, t(rt), t(offs), k, K, t(qbar), t(vbar), t(w1), t(b1.float()), t(w2.float()), b2)
        skip.skip_retrieve_skv(*args)
        assert skip.skip_sync_status(c) == skip.SKIP_ETIMEOUT
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        c.set_option(skip.SKIP_OPT_WAIT_TIMEOUT_NS, 2_000_000_000)
        g_ids, g_nu, g_cnt, m_ids, _ = skip.skip_retrieve_skv(*args, with_merged=True)
        ids_all = skip.skip_skv_gate(c, m_ids, t(qbar), t(vbar), t(w1), t(b1.float()), t(w2.float()), b2,
                                     with_nu_all=True)
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        for a, b in zip((g_ids, g_nu, g_cnt), ids_all[:3]):
            assert torch.equal(a, b)
        gpu = [x.cpu().numpy() for x in ids_all]
        mids = m_ids.cpu()
    finally:
        c.free()
    b = synth.bf16_bits
    o = oracle.skv(b(ct), mids.numpy(), b(qbar), b(vbar), b(w1), b1.float().numpy(), w2.float().numpy(), b2,
                   tau=0.5, rho=0.6)
    check_gate(gpu, o, mids, 0.5, 0.6)
