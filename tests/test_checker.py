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
    oid, osc = oracle.merge(ids, sc, k, offsets, K + 1)
    return cb, qb, ids, sc, oid, osc, offsets, k, K


def _question(cb, qb, ids, sc, oid, osc, offsets, k, K, q, g, s, lists=None):
    truths = checker.region_truths(ids, sc, k)
    r0, r1 = offsets[q], offsets[q + 1]
    ts = truths[r0:r1]
    rescore = checker.exact_rescore(cb, qb[r0:r1], ts)
    if lists is None:
        lists = ids[r0:r1, :k]
    return checker.check_question(g, s, oid[q], osc[q], ts, K, lists, rescore)


def test_oracle_output_passes():
    cb, qb, ids, sc, oid, osc, offsets, k, K = _truth()
    truths = checker.region_truths(ids, sc, k)
    for r, t in enumerate(truths):
        ex, pr = checker.check_region(ids[r, :k], sc[r, :k].astype(np.float32), t)
        assert ex and not pr
    for q in range(2):
        ex, pr, _ = _question(cb, qb, ids, sc, oid, osc, offsets, k, K, q, oid[q, :K],
                              osc[q, :K].astype(np.float32))
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
    args = _truth(2)
    cb, qb, ids, sc, oid, osc, offsets, k, K = args
    g, s = oid[0, :K].copy(), osc[0, :K].astype(np.float32)
    # Lost id: drop the best and shift.
    g2 = np.concatenate([g[1:], [-1]]); s2 = np.concatenate([s[1:], [-math.inf]]).astype(np.float32)
    assert _question(*args, 0, g2, s2)[1]
    # Duplicate instead of dedup.
    g3 = g.copy(); g3[2] = g3[1]
    assert _question(*args, 0, g3, s)[1]
    # Min score kept for a duplicate id: lower the score of a shared id well below.
    s4 = s.copy(); s4[0] -= 0.05
    assert _question(*args, 0, g, s4)[1]
    # Padding before a valid entry.
    g5 = g.copy(); g5[3] = -1
    assert _question(*args, 0, g5, s)[1]


# Three regions, k = 3, K = 4, tau = 2e-3; the scores are chosen by hand.
# Region 2's ranks 3 and 4 are 1e-4 apart (its band holds ids 11-14), but
# its 3rd score plus tau stays below the merged 4th score, so it cannot move
# the merged list: the question is unambiguous.
HAND_IDS = np.array([[1, 2, 3, 4, 5], [6, 7, 8, 9, 10], [11, 12, 13, 14, 15]], np.int64)
HAND_SC = np.array([[.950, .9485, .948, .900, .850], [.947, .930, .920, .880, .870],
                    [.9445, .9440, .9435, .9434, .800]])


def _hand(k=3, K=4, region2=(11, 12, 13), sc=HAND_SC):
    truths = checker.region_truths(HAND_IDS, sc, k)
    oid, osc = oracle.merge(HAND_IDS, sc, k, np.array([0, 3], np.int32), K + 1)
    table = {(j, int(i)): float(s) for j in range(3) for i, s in zip(HAND_IDS[j], sc[j])}

    def rescore(j, ids):
        return np.array([table[(j, int(i))] for i in ids])
    lists = [HAND_IDS[0, :k], HAND_IDS[1, :k], np.array(region2, np.int64)]
    return truths, oid[0], osc[0], lists, rescore


def test_mid_rank_swap_is_caught():
    """Dropping the rank-2 id and taking region 2's 4th-ranked id (in its
    near-tie band, so the per-region check alone would allow it) keeps every
    rank-wise score within 2 tau of the oracle's and leaves out no id that
    clears the last score by 2 tau; the question is unambiguous, so its id set
    must equal the oracle's."""
    truths, oid, osc, lists, rescore = _hand(region2=(11, 12, 14))
    assert list(oid[:4]) == [1, 2, 3, 6]
    good = checker.check_question(oid[:4], osc[:4], oid, osc, truths, 4, lists, rescore)
    assert good[0] and not good[1] and not good[2]
    g = np.array([1, 3, 6, 14])
    s = np.array([.950, .948, .947, .9434], np.float32)
    exact, probs, amb = checker.check_question(g, s, oid, osc, truths, 4, lists, rescore)
    assert probs and not exact and not amb
    assert "differs from the oracle's" in probs[0]


def test_ambiguous_question_follows_the_gpu_region_lists():
    """When a contributing region has a near-tie at its k-th rank, the GPU's
    region list may hold either tied id; the merged list must then be the
    oracle's merge of the GPU's own region lists, and nothing else."""
    sc = HAND_SC.copy()
    sc[2] = [.9475, .9472, .9471, .9470, .800]   # region 2 now reaches the merged top 4
    truths, oid, osc, _, rescore = _hand(sc=sc)
    lists = [HAND_IDS[0, :3], HAND_IDS[1, :3], np.array([11, 12, 14])]   # 14 instead of 13: a band choice
    m_ids, m_sc = oracle.merge(np.stack(lists), np.stack([rescore(j, x) for j, x in enumerate(lists)]), 3,
                               np.array([0, 3], np.int32), 5)
    g, s = m_ids[0, :4], m_sc[0, :4].astype(np.float32)
    exact, probs, amb = checker.check_question(g, s, oid, osc, truths, 4, lists, rescore)
    assert amb and not probs
    # An id of the GPU's region lists that its merge leaves out is refused.
    g2 = g.copy(); g2[1] = 8
    s2 = s.copy(); s2[1] = np.float32(.92)
    order = np.lexsort((g2, -s2.astype(np.float64)))
    assert checker.check_question(g2[order], s2[order], oid, osc, truths, 4, lists, rescore)[1]
