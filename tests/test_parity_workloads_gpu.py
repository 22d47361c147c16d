"""GPU parity at the full sizes of the five workloads, in the launch
configuration bench.py times (library defaults).

The whole batch runs on the GPU; the oracle then recomputes, by a full scan
of the corpus, the exact lists of a sample of questions (every region of each
sampled question) and the checker compares them (tests/checker.py): per
region, every sure id present and the rest from the near-tie band, scores
within 2e-3; per question, the deduplicated top-K.  Inputs are drawn on the
GPU with the workload's seeds and copied to the host for the oracle.
"""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2607_25422_gb300 as skip
import synth
from tests import checker

pytestmark = pytest.mark.gpu

# workload -> (questions to check, oracle extension past rank k)
SAMPLES = {
    "tiny_100k": ("all", 32),
    "clustered_1m": (16, 160),
    "throughput_10m": (16, 160),
    "latency_fp8_6m": ("all", 32),
    "ragged_20m": (8, 160),
}

# Floors on the strict exact-match rates (ids in the oracle's order, scores
# within 2e-3, no near-tie excuse), per region list and per question: the
# GPU sums in fp32 (~1e-6 from the fp64 value), so a list differs from the
# oracle's only where two of its scores lie closer than that, which
# clustered corpora with k = 100 make common; the small-batch e4m3 path's
# three-part queries (within 2.4e-4 of exact) could reorder more, and its
# single question is reported, not required.  Measured rates are printed
# (at the time of writing 1.0 / 1.0, 1.0 / 0.94, 0.98 / 0.88, 1.0 / 1.0 and
# 0.84 / 1.0).
STRICT_FLOOR = {
    "tiny_100k": (1.0, 1.0),
    "clustered_1m": (0.95, 0.8),
    "throughput_10m": (0.9, 0.75),
    "latency_fp8_6m": (0.9, 0.0),
    "ragged_20m": (0.75, 0.75),
}


def _pick_questions(offsets, how):
    """All questions, or `how` of them drawn with a fixed seed, always
    including a question with the fewest and one with the most regions."""
    counts = np.diff(offsets)
    Q = counts.size
    if how == "all":
        return list(range(Q))
    keep = {int(np.argmin(counts)), int(np.argmax(counts))}
    rng = np.random.default_rng(12345)
    for q in rng.permutation(Q).tolist():
        if len(keep) >= how:
            break
        keep.add(int(q))
    return sorted(keep)


@pytest.mark.parametrize("name", list(SAMPLES))
def test_workload_full_size(name):
    spec = synth.WORKLOADS[name]
    how, extra = SAMPLES[name]
    dev = torch.device("cuda")
    corpus, scale, centres = synth.make_corpus(spec, device=dev)
    regions, offsets = synth.make_regions(spec, centres, "cpu")
    c = skip.skip_corpus_load(corpus, row_scale=scale)
    try:
        reg_d, off_d = regions.to(dev), offsets.to(dev)
        rid, rsc = skip.skip_retrieve_regions(c, reg_d, spec.k_region)
        oid, osc = skip.skip_retrieve(c, reg_d, off_d, spec.k_region, spec.K)
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        plan = skip.skip_last_plan(c)
        rid, rsc, oid, osc = (t.cpu().numpy() for t in (rid, rsc, oid, osc))
    finally:
        c.free()
    if spec.dtype == "bf16":
        cn, sn = synth.bf16_bits(corpus), None
    else:
        cn, sn = corpus.cpu().numpy(), scale.cpu().numpy()
    del corpus
    torch.cuda.empty_cache()
    off = offsets.numpy()
    qs = _pick_questions(off, how)
    rows = [r for q in qs for r in range(off[q], off[q + 1])]
    rn = synth.bf16_bits(regions[rows])
    kk = min(spec.N, spec.k_region + extra)
    ids_ext, sc_ext = oracle.region_topk(cn, rn, kk, row_scale=sn, nthreads=len(os.sched_getaffinity(0)))
    truths = checker.region_truths(ids_ext, sc_ext, spec.k_region)
    bad = []
    exact = 0
    for t, r in zip(truths, rows):
        ex, probs = checker.check_region(
            rid[r], rsc[r], t,
            extra_score=lambda i, r=r: float(oracle.scores_at(cn, synth.bf16_bits(regions[r:r + 1]), [0], [i],
                                                               row_scale=sn)[0]))
        exact += ex
        if probs:
            bad.append(("region", r, probs[:3]))
    at = 0
    q_exact = q_amb = 0
    for q in qs:
        n = off[q + 1] - off[q]
        ts = truths[at:at + n]
        sub_ids, sub_sc = ids_ext[at:at + n], sc_ext[at:at + n]
        sub_rn = rn[at:at + n]
        at += n
        o_ids, o_sc = oracle.merge(sub_ids, sub_sc, spec.k_region, np.array([0, n], np.int32), spec.K + 1)
        rescore = checker.exact_rescore(cn, sub_rn, ts, row_scale=sn)
        ex, probs, amb = checker.check_question(oid[q], osc[q], o_ids[0], o_sc[0], ts, spec.K,
                                                rid[off[q]:off[q + 1]], rescore)
        q_exact += ex
        q_amb += amb
        if probs:
            bad.append(("question", q, probs[:3]))
    assert not bad, "%s plan %s: %s" % (name, plan, bad[:5])
    r_rate, q_rate = exact / len(rows), q_exact / len(qs)
    print("%s: strict exact match %d of %d region lists (%.3f), %d of %d questions (%.3f); "
          "%d questions near-tied" % (name, exact, len(rows), r_rate, q_exact, len(qs), q_rate, q_amb))
    lo_r, lo_q = STRICT_FLOOR[name]
    assert r_rate >= lo_r and q_rate >= lo_q, (r_rate, q_rate)
