"""Tolerance-aware comparison of the CUDA path's lists with the oracle's.

Tolerance: |score_gpu - score_oracle| <= TAU (2e-3) for unit-norm inputs; id
sets must match except where the oracle's ranks k and k + 1 differ by less
than TAU.  The GPU accumulates in fp32 (error ~1e-6), so almost every list
matches exactly; the band rules only excuse near-ties.

Per region (oracle list extended past rank k):
  theta = oracle k-th score; sure = {s > theta + TAU}; band = {|s - theta| <= TAU}.
  The GPU list must hold every sure id, draw its other ids from the band,
  and report every score within TAU of the oracle's fp64 value.
Per question (the GPU's per-region lists of its regions have passed the
per-region check):
  * ids unique, padding (-1, -inf) only at the tail, sorted by
    (score desc, id asc);
  * each score within TAU of the fp64 maximum of s(r, id) over the
    question's regions r whose GPU list holds the id (an id in none of them
    is an error);
  * unambiguous question -- the oracle's merged rank-K / K+1 scores differ
    by at least TAU (or the union has at most K ids) and no contributing
    region (one whose k-th score is within TAU of the merged K-th score or
    above it) has its k / k+1 scores closer than TAU: the GPU id set equals
    the oracle's;
  * otherwise the oracle's merge (step 4, Dedup of the union) is run again
    on the GPU's own per-region lists, re-scored in fp64 by the oracle, and
    the GPU id set must equal that merge's (up to its own rank-K / K+1 band
    when those differ by less than TAU).
  * strict (reported, not required): ids equal the oracle's in order and
    scores within TAU.
"""
from __future__ import annotations

import math

import numpy as np

TAU = 2e-3


class RegionTruth:
    """Oracle view of one region: its exact list extended past rank k."""

    def __init__(self, ids, scores, k, tau=TAU):
        self.k = k
        self.ids = [int(i) for i in ids if i >= 0]
        self.scores = [float(s) for i, s in zip(ids, scores) if i >= 0]
        self.score_of = dict(zip(self.ids, self.scores))
        self.theta = self.scores[k - 1]
        self.sure = {i for i, s in zip(self.ids, self.scores) if s > self.theta + tau}
        self.band = {i for i, s in zip(self.ids, self.scores) if abs(s - self.theta) <= tau}
        # The extended list is long enough when it reaches below the band.
        self.complete = len(self.ids) < len(ids) or self.scores[-1] < self.theta - tau


def check_region(gpu_ids, gpu_scores, truth: RegionTruth, extra_score=None, tau=TAU):
    """Returns (exact, problems). extra_score(id) gives the oracle's score of
    an id outside the extended list (or None)."""
    problems = []
    g = [int(i) for i in gpu_ids]
    gs = [float(s) for s in gpu_scores]
    k = truth.k
    if len(g) != k or len(set(g)) != k or min(g) < 0:
        problems.append("ids not %d distinct valid ids: %s" % (k, g[:8]))
        return False, problems
    missing = truth.sure - set(g)
    if missing:
        problems.append("sure ids missing: %s" % sorted(missing)[:8])
    for i, s in zip(g, gs):
        if i in truth.score_of:
            ref = truth.score_of[i]
            if i not in truth.sure and i not in truth.band:
                problems.append("id %d outside the band (s=%.6f theta=%.6f)" % (i, ref, truth.theta))
        else:
            ref = extra_score(i) if extra_score else None
            if ref is None or abs(ref - truth.theta) > tau:
                problems.append("id %d not in the oracle list (s=%s)" % (i, ref))
                continue
        if abs(s - ref) > tau:
            problems.append("id %d score %.7f vs oracle %.7f" % (i, s, ref))
    for a, b, ia, ib in zip(gs, gs[1:], g, g[1:]):
        if a < b or (a == b and ia > ib):
            problems.append("list not sorted by (score desc, id asc)")
            break
    exact = not problems and g == truth.ids[:k]
    return exact, problems


def _gap_at(scores, k):
    """Score at rank k minus the score at rank k + 1 (1-based ranks), inf
    when rank k + 1 is absent or padding."""
    if len(scores) <= k or not math.isfinite(scores[k]):
        return math.inf
    return scores[k - 1] - scores[k]


def check_question(gpu_ids, gpu_scores, ora_ids, ora_scores, truths, K, gpu_lists, rescore, tau=TAU):
    """One question.

    ora_ids, ora_scores -- the oracle's merged list, at least K + 1 slots long
        (oracle.merge(..., K + 1)): slot K + 1 gives the merged K / K+1 gap.
    truths -- RegionTruth of each of the question's regions.
    gpu_lists -- the GPU's per-region id lists of the same regions.
    rescore(j, ids) -- the oracle's fp64 scores of `ids` for region j.
    Returns (exact, problems, ambiguous)."""
    import oracle

    g = [int(i) for i in gpu_ids]
    gs = [float(s) for s in gpu_scores]
    o = [int(i) for i in ora_ids]
    os_ = [float(s) for s in ora_scores]
    if len(o) < K + 1:
        raise ValueError("the oracle's merged list must hold K + 1 slots")
    nval = sum(1 for i in g if i >= 0)
    if any(i < 0 for i in g[:nval]) or any(i >= 0 for i in g[nval:]):
        return False, ["padding not at the tail"], False
    if any(not (math.isinf(s) and s < 0) for s in gs[nval:]):
        return False, ["padding scores not -inf"], False
    problems = []
    valid = g[:nval]
    if len(set(valid)) != nval:
        problems.append("duplicate ids")
    for a, b, ia, ib in zip(gs[:nval], gs[1:nval], valid, valid[1:]):
        if a < b or (a == b and ia > ib):
            problems.append("list not sorted by (score desc, id asc)")
            break
    # Scores: the max over the regions whose GPU list holds the id.
    lists = [np.asarray(x, dtype=np.int64) for x in gpu_lists]
    fresh = [rescore(j, x[x >= 0]) if (x >= 0).any() else np.zeros(0) for j, x in enumerate(lists)]
    best = {}
    for x, sc in zip(lists, fresh):
        for i, v in zip(x[x >= 0].tolist(), np.asarray(sc, dtype=np.float64).tolist()):
            best[i] = max(best.get(i, -math.inf), v)
    for i, s in zip(valid, gs):
        if i not in best:
            problems.append("id %d in none of the question's GPU region lists" % i)
        elif abs(s - best[i]) > tau:
            problems.append("id %d score %.7f vs oracle max %.7f" % (i, s, best[i]))
    onval = sum(1 for i in o[:K] if i >= 0)
    exact = not problems and g == o[:K] and all(abs(a - b) <= tau for a, b in zip(gs[:nval], os_[:nval]))
    oK = os_[K - 1] if o[K - 1] >= 0 else -math.inf
    merged_amb = _gap_at(os_, K) < tau
    region_amb = any(_gap_at(t.scores, t.k) < tau and t.theta + tau >= oK for t in truths)
    ambiguous = merged_amb or region_amb
    if not ambiguous:
        if set(valid) != set(o[:onval]) or nval != onval:
            problems.append("id set differs from the oracle's (no near-tie excuses it): extra %s, missing %s"
                            % (sorted(set(valid) - set(o[:onval]))[:6], sorted(set(o[:onval]) - set(valid))[:6]))
        return exact, problems, False
    # Near-ties: the oracle's Dedup step on the GPU's own region lists.
    if lists:
        k = max(len(x) for x in lists)
        ids = np.full((len(lists), k), -1, np.int64)
        scs = np.full((len(lists), k), -math.inf)
        for j, (x, sc) in enumerate(zip(lists, fresh)):
            m = x >= 0
            ids[j, :m.sum()] = x[m]
            scs[j, :m.sum()] = sc
        m_ids, m_sc = oracle.merge(ids, scs, k, np.array([0, len(lists)], np.int32), K + 1)
        m_ids, m_sc = m_ids[0].tolist(), m_sc[0].tolist()
    else:
        m_ids, m_sc = [-1] * (K + 1), [-math.inf] * (K + 1)
    mval = sum(1 for i in m_ids[:K] if i >= 0)
    if _gap_at(m_sc, K) >= tau:
        if set(valid) != set(m_ids[:mval]) or nval != mval:
            problems.append("id set differs from the oracle's merge of the GPU's region lists: extra %s, missing %s"
                            % (sorted(set(valid) - set(m_ids[:mval]))[:6], sorted(set(m_ids[:mval]) - set(valid))[:6]))
    else:
        theta = m_sc[K - 1]
        sure = {i for i, s in zip(m_ids, m_sc) if i >= 0 and s > theta + tau}
        band = {i for i, s in zip(m_ids, m_sc) if i >= 0 and abs(s - theta) <= tau}
        if not sure <= set(valid):
            problems.append("merge of the GPU's region lists: sure ids missing %s" % sorted(sure - set(valid))[:6])
        if not set(valid) <= sure | band:
            problems.append("merge of the GPU's region lists: ids outside its band %s"
                            % sorted(set(valid) - sure - band)[:6])
        if nval != mval:
            problems.append("%d entries, the merge of the GPU's region lists has %d" % (nval, mval))
    return exact, problems, True


def exact_rescore(corpus, regions_of_q, truths, row_scale=None):
    """rescore(j, ids) for the exact path: the oracle's fp64 s(r_j, id), from
    the extended list where it holds the id, else computed."""
    import oracle

    def rescore(j, ids):
        ids = np.asarray(ids, dtype=np.int64)
        out = np.array([truths[j].score_of.get(int(i), math.nan) for i in ids], dtype=np.float64)
        miss = np.isnan(out)
        if miss.any():
            out[miss] = oracle.scores_at(corpus, regions_of_q, np.full(int(miss.sum()), j), ids[miss],
                                         row_scale=row_scale)
        return out
    return rescore


def region_truths(ora_ids_ext, ora_scores_ext, k, tau=TAU):
    return [RegionTruth(a, b, k, tau) for a, b in zip(ora_ids_ext, ora_scores_ext)]
