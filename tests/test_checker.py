"""The parity checker catches mistakes planted in the oracle's own output."""
import math

import numpy as np

import oracle
import synth
from tests import checker


def _truth(seed=0, N=3000, d=64, R=4, k=8, K=12):
    cb = synth.bf16_bits(synth.random_bf16(N, d, seed))
    qb = synth.bf16_bits(synth.random_bf16(R, d, seed + 1))
    ids, sc = oracle.region_topk(cb, qb, k + 40)
    offsets = np.array([0, 2, R], np.int32)
    oid, osc = oracle.merge(ids, sc, k, offsets, K)
    return cb, qb, ids, sc, oid, osc, offsets, k, K


def test_oracle_output_passes():
    cb, qb, ids, sc, oid, osc, offsets, k, K = _truth()
    truths = checker.region_truths(ids, sc, k)
    for r, t in enumerate(truths):
        ex, pr = checker.check_region(ids[r, :k], sc[r, :k].astype(np.float32), t)
        assert ex and not pr
    for q in range(2):
        ex, pr = checker.check_question(oid[q], osc[q].astype(np.float32), oid[q], osc[q],
                                        truths[offsets[q]:offsets[q + 1]], K)
        assert ex and not pr


def test_planted_region_mistakes_are_caught():
    cb, qb, ids, sc, *_ , k, K = _truth(1)
    t = checker.RegionTruth(ids[0], sc[0], k)
    g, s = ids[0, :k].copy(), sc[0, :k].astype(np.float32)
    # A dropped top id replaced by rank k + 20 (far below the band).
    g2 = g.copy(); g2[0] = ids[0, k + 20]
    assert checker.check_region(g2, s, t)[1]
    # A score off by 1e-2.
    s2 = s.copy(); s2[3] += 1e-2
    assert checker.check_region(g, s2, t)[1]
    # Reversed order.
    assert checker.check_region(g[::-1], s[::-1], t)[1]
    # Duplicate id.
    g3 = g.copy(); g3[1] = g3[0]
    assert checker.check_region(g3, s, t)[1]


def test_planted_merge_mistakes_are_caught():
    cb, qb, ids, sc, oid, osc, offsets, k, K = _truth(2)
    truths = checker.region_truths(ids, sc, k)[0:2]
    g, s = oid[0].copy(), osc[0].astype(np.float32)
    # Lost id: drop the best and shift.
    g2 = np.concatenate([g[1:], [-1]]); s2 = np.concatenate([s[1:], [-math.inf]]).astype(np.float32)
    assert checker.check_question(g2, s2, oid[0], osc[0], truths, K)[1]
    # Duplicate instead of dedup.
    g3 = g.copy(); g3[2] = g3[1]
    assert checker.check_question(g3, s, oid[0], osc[0], truths, K)[1]
    # Min score kept for a duplicate id: lower the score of a shared id well below.
    s4 = s.copy(); s4[0] -= 0.05
    assert checker.check_question(g, s4, oid[0], osc[0], truths, K)[1]
