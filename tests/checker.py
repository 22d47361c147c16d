"""Tolerance-aware comparison of the CUDA path's lists with the oracle's.

Tolerance: |score_gpu - score_oracle| <= TAU (2e-3) for unit-norm inputs; id
sets must match except where the oracle's ranks k and k + 1 differ by less
than TAU.  The GPU accumulates in fp32 (error ~1e-6), so almost every list
matches exactly; the band rules only excuse near-ties.

Per region (oracle list extended past rank k):
  theta = oracle k-th score; sure = {s > theta + TAU}; band = {|s - theta| <= TAU}.
  The GPU list must hold every sure id, draw its other ids from the band,
  and report every score within TAU of the oracle's fp64 value.
Per question:
  strict -- ids equal the oracle's and scores within TAU; otherwise
  tolerant -- ids unique and admissible (sure or band in one of the
  question's regions), each score between the id's sure-region maximum and
  its admissible-region maximum (each +- TAU), rank-wise scores within
  2 TAU of the oracle's, and no id whose sure score clears the GPU's last
  score by 2 TAU left out.
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


def check_question(gpu_ids, gpu_scores, ora_ids, ora_scores, truths, K, tau=TAU):
    """truths: RegionTruth of each of the question's regions."""
    g = [int(i) for i in gpu_ids]
    gs = [float(s) for s in gpu_scores]
    o = [int(i) for i in ora_ids]
    os_ = [float(s) for s in ora_scores]
    nval = sum(1 for i in g if i >= 0)
    if any(i < 0 for i in g[:nval]) or any(i >= 0 for i in g[nval:]):
        return False, ["padding not at the tail"]
    if any(not (math.isinf(s) and s < 0) for s in gs[nval:]):
        return False, ["padding scores not -inf"]
    if g == o and all(abs(a - b) <= tau for a, b in zip(gs[:nval], os_[:nval])):
        return True, []
    problems = []
    valid = g[:nval]
    if len(set(valid)) != nval:
        problems.append("duplicate ids")
    lo, hi = {}, {}
    for t in truths:
        for i, s in t.score_of.items():
            if i in t.sure:
                lo[i] = max(lo.get(i, -math.inf), s)
            if i in t.sure or i in t.band:
                hi[i] = max(hi.get(i, -math.inf), s)
    for i, s in zip(valid, gs):
        if i not in hi:
            problems.append("id %d not admissible" % i)
        elif s < lo.get(i, -math.inf) - tau or s > hi[i] + tau:
            problems.append("id %d score %.6f outside [%.6f, %.6f]" % (i, s, lo.get(i, -math.inf), hi[i]))
    onval = sum(1 for i in o if i >= 0)
    for p in range(min(nval, onval)):
        if abs(gs[p] - os_[p]) > 2 * tau:
            problems.append("rank %d score %.6f vs oracle %.6f" % (p, gs[p], os_[p]))
            break
    if nval == K:
        last = gs[nval - 1]
        for i, s in lo.items():
            if s > last + 2 * tau and i not in set(valid):
                problems.append("id %d (sure score %.6f) left out" % (i, s))
                break
    elif nval < min(K, len(lo)):
        problems.append("only %d entries, %d sure candidates" % (nval, len(lo)))
    return False, problems


def region_truths(ora_ids_ext, ora_scores_ext, k, tau=TAU):
    return [RegionTruth(a, b, k, tau) for a, b in zip(ora_ids_ext, ora_scores_ext)]
