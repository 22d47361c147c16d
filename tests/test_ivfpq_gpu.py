"""GPU parity of the IVF-PQ variant (inverted file over inner-product
centroids, product-quantised residual codes, asymmetric scoring; the index
of §4.1 "Implementation" / App. I.4) against the oracle
(oracle/ivfpq_oracle.c).

* Build: the GPU's lists and codes equal the oracle's, except where the
  oracle's own values show a near tie (the two centroid scores, or the two
  codeword distances, within fp32 rounding of each other).
* Search: on the oracle's index loaded into the GPU, per-region lists are
  checked as the exact path's are (tests/checker.py: sure ids present, the
  rest from the 2e-3 band, scores within 2e-3 of the oracle's s^), skipping
  regions whose nprobe-th and next centroid scores are within PROBE_TIE
  (there the probed lists themselves may differ: the GPU's centroid scores
  are fp32 sums of 2d bf16 products, off by ~1e-6); merged lists per
  question likewise.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_25422_gb300 as skip
import synth
from tests import checker
from tests._golden import read_fixture

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")
PROBE_TIE = 1e-4


def _t(x, dtype=None):
    x = torch.as_tensor(x)
    return (x if dtype is None else x.to(dtype)).to(DEV).contiguous()


def _embed_hand():
    """The hand example of tests/golden/ivfpq_hand_example.txt in d = 64,
    M = 16 (sub-space width 4): hand sub-space 0 -> dims 0-1, hand sub-space
    1 -> dims 4-5, every other coordinate 0; codewords 2..255 far away."""
    fx = read_fixture("ivfpq_hand_example.txt")
    d, M, ds = 64, 16, 4
    place = [0, 1, 4, 5]

    def emb(rows):
        out = np.zeros((rows.shape[0], d), np.float32)
        out[:, place] = rows
        return out
    cb = np.full((M, 256, ds), 100.0, np.float32)
    cb[:, :2] = 0.0
    hcb = fx["codebook"].reshape(2, 2, 2)
    for m in range(2):
        cb[m, :2, :2] = hcb[m]
    return fx, emb(fx["ivf_corpus"]), emb(fx["centroids"]), emb(fx["queries"]), cb


def test_hand_example_build_and_search():
    fx, corpus, cent, q, cb = _embed_hand()
    bf = lambda a: torch.from_numpy(a).to(torch.bfloat16)
    c = skip.skip_corpus_load(_t(bf(corpus)))
    try:
        ix = skip.skip_ivfpq_build(c, _t(bf(cent)), _t(cb))
        off, ids, codes = (x.cpu().numpy() for x in skip.skip_ivfpq_lists(ix))
        lists = np.empty(ix.N, np.int32)
        code_by_id = np.empty((ix.N, ix.M), np.uint8)
        for l in range(ix.C):
            lists[ids[off[l]:off[l + 1]]] = l
            code_by_id[ids[off[l]:off[l + 1]]] = codes[off[l]:off[l + 1]]
        np.testing.assert_array_equal(lists, fx["lists"].astype(np.int32))
        np.testing.assert_array_equal(code_by_id[:, :2], fx["codes"].astype(np.uint8))
        assert np.all(code_by_id[:, 2:] == 0)
        for p, k, key in ((1, 2, "p1k2"), (1, 4, "p1k4"), (2, 3, "p2k3")):
            g_ids, g_sc = skip.skip_ivfpq_search_regions(ix, _t(bf(q)), p, k)
            assert skip.skip_ivfpq_sync_status(ix) == skip.SKIP_OK
            np.testing.assert_array_equal(g_ids.cpu().numpy(), fx[key + "_ids"].astype(np.int64))
            np.testing.assert_array_equal(g_sc.cpu().numpy(), fx[key + "_scores"].astype(np.float32))
        ix.free()
    finally:
        c.free()


SPEC = synth.WorkloadSpec("ivf_small", 41, 30000, 128, "bf16", 12, (1, 8), 10, 25, "clustered", 64)


def _small_inputs(M=16):
    corpus, _, centres = synth.make_corpus(SPEC)
    regions, offsets = synth.make_regions(SPEC, centres)
    cent = synth.make_ivf_centroids(SPEC)
    cb = synth.make_pq_codebook(SPEC, M)
    return corpus, regions, offsets, cent, cb


def _lists_by_id(off, ids, codes, N, M):
    lists = np.full(N, -1, np.int32)
    code_by_id = np.zeros((N, M), np.uint8)
    for l in range(off.shape[0] - 1):
        lists[ids[off[l]:off[l + 1]]] = l
        code_by_id[ids[off[l]:off[l + 1]]] = codes[off[l]:off[l + 1]]
    return lists, code_by_id


def check_build(corpus, cent, cb, lists, code_by_id, rows):
    """GPU lists/codes of the given rows against the oracle's, near ties aside."""
    cn, ce = synth.bf16_bits(corpus[rows]), synth.bf16_bits(cent)
    o_lists = oracle.ivf_assign(cn, ce)
    s = oracle.score_matrix(ce, cn)  # [n, C] exact centroid scores
    n_diff_list = n_diff_code = 0
    for t, i in enumerate(rows):
        if lists[i] != o_lists[t]:
            n_diff_list += 1
            assert abs(s[t, lists[i]] - s[t, o_lists[t]]) <= 1e-5, (i, lists[i], o_lists[t])
    same = [t for t, i in enumerate(rows) if lists[i] == o_lists[t]]
    o_codes = oracle.pq_encode(cn[same], ce, o_lists[same], cb)
    x = corpus[rows].double().numpy()[same]
    c = cent.double().numpy()[o_lists[same]]
    ds = cb.shape[2]
    for m in range(cb.shape[0]):
        g = code_by_id[np.asarray(rows)[same], m]
        bad = np.nonzero(g != o_codes[:, m])[0]
        for b in bad:
            r = x[b, m * ds:(m + 1) * ds] - c[b, m * ds:(m + 1) * ds]
            dist = ((r[None, :] - cb[m].double().numpy()) ** 2).sum(1)
            assert dist[g[b]] - dist[o_codes[b, m]] <= 1e-6 * max(1.0, dist.max()), (b, m)
        n_diff_code += len(bad)
    return n_diff_list, n_diff_code


def test_build_matches_oracle():
    corpus, regions, offsets, cent, cb = _small_inputs()
    c = skip.skip_corpus_load(_t(corpus))
    try:
        ix = skip.skip_ivfpq_build(c, _t(cent), _t(cb))
        off, ids, codes = (x.cpu().numpy() for x in skip.skip_ivfpq_lists(ix))
        ix.free()
    finally:
        c.free()
    assert off[-1] == SPEC.N and sorted(ids.tolist()) == list(range(SPEC.N))
    lists, code_by_id = _lists_by_id(off, ids, codes, SPEC.N, cb.shape[0])
    nl, nc = check_build(corpus, cent, cb, lists, code_by_id, list(range(SPEC.N)))
    print("build: %d list and %d code differences from the oracle, all near ties" % (nl, nc))


@pytest.mark.parametrize("nprobe", [1, 4, 16, 64])
def test_search_matches_oracle(nprobe):
    _check_search(SPEC, 16, nprobe)


@pytest.mark.parametrize("d,M", [(128, 32), (96, 48), (160, 80), (128, 128)])
def test_search_sub_space_counts(d, M):
    """One to four warps' worth of sub-spaces (the lookup table's row is M
    rounded up to 32), including the half-warp passes of M = 48 and 80."""
    spec = synth.WorkloadSpec("ivf_m%d" % M, 43 + M, 9000, d, "bf16", 10, (1, 6), 10, 25, "clustered", 64)
    _check_search(spec, M, 8)


def _check_search(spec, M, nprobe):
    corpus, _, centres = synth.make_corpus(spec)
    regions, offsets = synth.make_regions(spec, centres)
    cent = synth.make_ivf_centroids(spec)
    cb = synth.make_pq_codebook(spec, M)
    cn, ce, qn = synth.bf16_bits(corpus), synth.bf16_bits(cent), synth.bf16_bits(regions)
    idx = oracle.ivfpq_build(cn, ce, cb.numpy())
    k, K = spec.k_region, spec.K
    ext = k + 32
    o_ids, o_sc, o_probes = oracle.ivfpq_search(idx, ce, cb.numpy(), qn, nprobe, ext)
    c = skip.skip_corpus_load(_t(corpus))
    try:
        ix = skip.skip_ivfpq_load(_t(cent), _t(cb), _t(idx["offsets"]), _t(idx["ids"], torch.int32),
                                  _t(idx["codes"][idx["ids"]]))
        g_ids, g_sc = skip.skip_ivfpq_search_regions(ix, _t(regions), nprobe, k)
        q_ids, q_sc = skip.skip_ivfpq_search(ix, _t(regions), _t(offsets), nprobe, k, K)
        assert skip.skip_ivfpq_sync_status(ix) == skip.SKIP_OK
        ix.free()
    finally:
        c.free()
    g_ids, g_sc, q_ids, q_sc = (x.cpu().numpy() for x in (g_ids, g_sc, q_ids, q_sc))
    cs = np.sort(oracle.score_matrix(ce, qn), axis=1)[:, ::-1]  # [R, C] centroid scores, descending
    truths = checker.region_truths(o_ids, o_sc, k)
    checked = exact = 0
    for r, t in enumerate(truths):
        if nprobe < cent.shape[0] and cs[r, nprobe - 1] - cs[r, nprobe] <= PROBE_TIE:
            continue  # the probed lists themselves are in the band
        ex, probs = checker.check_region(
            g_ids[r], g_sc[r], t,
            extra_score=lambda i, r=r: float(oracle.ivfpq_scores_at(idx, ce, cb.numpy(), qn, [r], [i])[0]))
        assert not probs, (r, probs[:3])
        checked += 1
        exact += ex
    assert checked >= len(truths) // 2
    off = offsets.numpy()
    o_m_ids, o_m_sc = oracle.merge(o_ids, o_sc, k, off, K + 1)
    for q in range(off.shape[0] - 1):
        rs = range(off[q], off[q + 1])
        if any(nprobe < cent.shape[0] and cs[r, nprobe - 1] - cs[r, nprobe] <= PROBE_TIE for r in rs):
            continue

        def rescore(j, ids, r0=off[q]):
            return oracle.ivfpq_scores_at(idx, ce, cb.numpy(), qn, np.full(len(ids), r0 + j), ids)
        _, probs, _ = checker.check_question(q_ids[q], q_sc[q], o_m_ids[q], o_m_sc[q], truths[off[q]:off[q + 1]],
                                             K, g_ids[off[q]:off[q + 1]], rescore)
        assert not probs, (q, probs[:3])
    print("nprobe %d: %d regions checked, %d identical to the oracle's" % (nprobe, checked, exact))


def test_split_parts_give_identical_lists():
    """Cutting each region's probed blocks into 1, 2, 3 or 8 parts (each part
    scanned by its own CTA, the parts' lists merged afterwards) changes
    nothing: every entry's s^ is computed the same way and ties break by id."""
    corpus, regions, offsets, cent, cb = _small_inputs()
    k, K = SPEC.k_region, SPEC.K
    c = skip.skip_corpus_load(_t(corpus))
    try:
        ix = skip.skip_ivfpq_build(c, _t(cent), _t(cb))
        outs = []
        for split in (1, 2, 3, 8, 0):
            ix.set_option(skip.SKIP_OPT_IVF_SPLIT, split)
            r_ids, r_sc = skip.skip_ivfpq_search_regions(ix, _t(regions), 16, k)
            q_ids, q_sc = skip.skip_ivfpq_search(ix, _t(regions), _t(offsets), 16, k, K)
            assert skip.skip_ivfpq_sync_status(ix) == skip.SKIP_OK
            outs.append([x.cpu().numpy() for x in (r_ids, r_sc, q_ids, q_sc)])
        with pytest.raises(skip.SkipError):
            ix.set_option(skip.SKIP_OPT_IVF_SPLIT, 9)
        ix.free()
    finally:
        c.free()
    for o in outs[1:]:
        for a, b in zip(outs[0], o):
            np.testing.assert_array_equal(a, b)


def test_ragged_lists_round_trip_and_search():
    """Lists of 0, 1, 31, 32, 33 and 100 entries (empty, partial and whole
    blocks of 32): the codes come back out of the index unchanged, a search
    probing every list returns the oracle's lists, and offsets that do not
    partition the N entries are refused."""
    rng = np.random.default_rng(11)
    gen = torch.Generator().manual_seed(11)
    lens = [0, 1, 31, 32, 33, 0, 100, 5]
    C, d, M = len(lens), 64, 32
    N = int(sum(lens))
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    ids = rng.permutation(N).astype(np.int64)
    lists = np.empty(N, np.int32)
    for l in range(C):
        lists[ids[off[l]:off[l + 1]]] = l
    codes_by_id = rng.integers(0, 256, (N, M), dtype=np.uint8)
    cent = torch.randn(C, d, generator=gen).to(torch.bfloat16)
    cb = torch.randn(M, 256, d // M, generator=gen) * 0.1
    q = torch.randn(6, d, generator=gen).to(torch.bfloat16)
    k = 40
    ix = skip.skip_ivfpq_load(_t(cent), _t(cb), _t(off), _t(ids, torch.int32), _t(codes_by_id[ids]))
    try:
        o, i, c = (x.cpu().numpy() for x in skip.skip_ivfpq_lists(ix))
        g_ids, g_sc = skip.skip_ivfpq_search_regions(ix, _t(q), C, k)
        assert skip.skip_ivfpq_sync_status(ix) == skip.SKIP_OK
    finally:
        ix.free()
    np.testing.assert_array_equal(o, off)
    np.testing.assert_array_equal(i, ids.astype(np.int32))
    np.testing.assert_array_equal(c, codes_by_id[ids])
    idx = {"offsets": off, "ids": ids, "codes": codes_by_id, "lists": lists}
    ce, qn = synth.bf16_bits(cent), synth.bf16_bits(q)
    o_ids, o_sc, _ = oracle.ivfpq_search(idx, ce, cb.numpy(), qn, C, k + 16)
    for r, t in enumerate(checker.region_truths(o_ids, o_sc, k)):
        _, probs = checker.check_region(
            g_ids[r].cpu().numpy(), g_sc[r].cpu().numpy(), t,
            extra_score=lambda i, r=r: float(oracle.ivfpq_scores_at(idx, ce, cb.numpy(), qn, [r], [i])[0]))
        assert not probs, (r, probs[:3])
    falling = off.copy()
    falling[4] = off[3] - 1
    for bad in (off + 1, np.r_[off[:-1], N - 1], falling):
        with pytest.raises(skip.SkipError):
            skip.skip_ivfpq_load(_t(cent), _t(cb), _t(bad), _t(ids, torch.int32), _t(codes_by_id[ids]))


def test_exact_codebook_all_lists_equals_exact_search():
    """With every residual sub-vector a codeword and every list probed, the
    IVF-PQ scores are the exact inner products: the GPU search must agree with
    the GPU's exact path (and the oracle's exact MIPS)."""
    spec = synth.WorkloadSpec("ivf_exact_gpu", 42, 256, 64, "bf16", 5, (2, 2), 8, 12, "clustered", 16)
    corpus, _, centres = synth.make_corpus(spec)
    regions, _ = synth.make_regions(spec, centres)
    cent = centres.to(torch.bfloat16)
    lists = oracle.ivf_assign(synth.bf16_bits(corpus), synth.bf16_bits(cent))
    M, ds = 16, 4
    r = (corpus.float() - cent.float()[torch.as_tensor(lists, dtype=torch.long)])
    cb = torch.stack([r[:, m * ds:(m + 1) * ds] for m in range(M)])
    c = skip.skip_corpus_load(_t(corpus))
    try:
        ix = skip.skip_ivfpq_build(c, _t(cent), _t(cb))
        g_ids, g_sc = skip.skip_ivfpq_search_regions(ix, _t(regions), spec.centres, spec.k_region)
        e_ids, e_sc = skip.skip_retrieve_regions(c, _t(regions), spec.k_region)
        assert skip.skip_ivfpq_sync_status(ix) == skip.SKIP_OK
        ix.free()
    finally:
        c.free()
    o_ids, o_sc = oracle.region_topk(synth.bf16_bits(corpus), synth.bf16_bits(regions), spec.k_region + 16)
    truths = checker.region_truths(o_ids, o_sc, spec.k_region)
    for rr, t in enumerate(truths):
        _, probs = checker.check_region(g_ids[rr].cpu().numpy(), g_sc[rr].cpu().numpy(), t)
        assert not probs, (rr, probs[:3])
    np.testing.assert_allclose(g_sc.cpu().numpy(), e_sc.cpu().numpy(), rtol=0, atol=1e-4)


def test_full_size_build_and_recall():
    """clustered_1m with the generator's 1,024 centres, PQ64 (sub-space width
    12) and 32 probes, in the configuration bench.py --ivfpq times.  Checked
    on sampled outputs the oracle computes one by one: sampled rows' lists
    and codes; for sampled regions, every returned id lies in a list the
    oracle would probe and its score equals the oracle's s^ for the oracle's
    own encoding of that row.  Recall@k against the exact path is reported
    (with these synthetic clusters the neighbours differ only by isotropic
    noise, which 8-bit codes of 12 values resolve poorly)."""
    spec = synth.WORKLOADS["clustered_1m"]
    nprobe = 32
    corpus, _, centres = synth.make_corpus(spec, device=DEV)
    regions, offsets = synth.make_regions(spec, centres, "cpu")
    cent = synth.make_ivf_centroids(spec)
    cb = synth.make_pq_codebook(spec, 64)
    c = skip.skip_corpus_load(corpus)
    try:
        ix = skip.skip_ivfpq_build(c, _t(cent), _t(cb))
        g_ids, g_sc = skip.skip_ivfpq_search_regions(ix, _t(regions), nprobe, spec.k_region)
        e_ids, _ = skip.skip_retrieve_regions(c, _t(regions), spec.k_region)
        assert skip.skip_ivfpq_sync_status(ix) == skip.SKIP_OK
        off, ids, codes = (x.cpu().numpy() for x in skip.skip_ivfpq_lists(ix))
        ix.free()
    finally:
        c.free()
    corpus = corpus.cpu()
    lists, code_by_id = _lists_by_id(off, ids, codes, spec.N, 64)
    rows = np.random.default_rng(7).choice(spec.N, 600, replace=False).tolist()
    nl, nc = check_build(corpus, cent, cb, lists, code_by_id, rows)
    g, gs, e = g_ids.cpu().numpy(), g_sc.cpu().numpy(), e_ids.cpu().numpy()
    ce, qn = synth.bf16_bits(cent), synth.bf16_bits(regions)
    # Completeness: the oracle's search of the GPU's own index (its lists and
    # codes, whose sampled rows match the oracle's encoding above) for the
    # sampled regions; every sure id of the oracle's list must be returned.
    gidx = {"offsets": off, "ids": ids.astype(np.int64), "codes": code_by_id, "lists": lists}
    sample = np.random.default_rng(8).choice(regions.shape[0], 6, replace=False)
    o_ids, o_sc, _ = oracle.ivfpq_search(gidx, ce, cb.numpy(), qn[sample], nprobe, spec.k_region + 32)
    complete = 0
    for j, t in enumerate(checker.region_truths(o_ids, o_sc, spec.k_region)):
        r = int(sample[j])
        cs = oracle.score_matrix(ce, qn[r:r + 1])[0]
        order = np.argsort(-cs, kind="stable")
        if cs[order[nprobe - 1]] - cs[order[nprobe]] <= PROBE_TIE:
            continue
        _, probs = checker.check_region(
            g_ids[r].cpu().numpy(), g_sc[r].cpu().numpy(), t,
            extra_score=lambda i, r=r: float(oracle.ivfpq_scores_at(gidx, ce, cb.numpy(), qn, [r], [i])[0]))
        assert not probs, (r, probs[:3])
        complete += 1
    assert complete >= 3
    checked = 0
    for r in sample:
        cs = oracle.score_matrix(ce, qn[r:r + 1])[0]
        order = np.argsort(-cs, kind="stable")
        if cs[order[nprobe - 1]] - cs[order[nprobe]] <= PROBE_TIE:
            continue
        probes = set(order[:nprobe].tolist())
        rid = g[r]
        rows_r = synth.bf16_bits(corpus[torch.as_tensor(rid)])
        o_list = oracle.ivf_assign(rows_r, ce)
        assert all(int(l) in probes for l in o_list), r
        o_code = oracle.pq_encode(rows_r, ce, o_list, cb.numpy())
        mini = {"lists": o_list, "codes": o_code}
        s_o = oracle.ivfpq_scores_at(mini, ce, cb.numpy(), qn, np.full(len(rid), r), np.arange(len(rid)))
        np.testing.assert_allclose(gs[r], s_o, rtol=0, atol=checker.TAU)
        assert np.all(np.diff(gs[r]) <= 0) and len(set(rid.tolist())) == len(rid)
        checked += 1
    assert checked >= 3
    recall = np.mean([len(set(a) & set(b)) / spec.k_region for a, b in zip(g, e)])
    print("clustered_1m IVF1024-PQ64, nprobe %d: recall@%d %.3f (random pick from the probed lists: %.4f); "
          "%d/%d sampled list/code differences (near ties)"
          % (nprobe, spec.k_region, recall, spec.k_region * spec.centres / (nprobe * spec.N), nl, nc))
    assert recall > 10 * spec.k_region * spec.centres / (nprobe * spec.N)


@pytest.mark.parametrize("refine", [2, 8])
def test_refine_matches_oracle(refine):
    """SKIP_OPT_IVF_REFINE = r: each region's best r k entries by s^ are
    re-scored exactly; the GPU's lists must pass the per-region check against
    the oracle's refined search (its shortlist re-ordered by exact fp64
    scores), and the per-question merge the question check.  Regions whose
    probed lists or whose shortlist end sit on a near tie in s^ (the GPU
    computes s^ in fp32) are left out.  An index made by skip_ivfpq_load has
    no corpus to re-rank against and refuses the option."""
    corpus, regions, offsets, cent, cb = _small_inputs()
    k, K, nprobe = SPEC.k_region, SPEC.K, 16
    ks = refine * k
    cn, ce, qn = synth.bf16_bits(corpus), synth.bf16_bits(cent), synth.bf16_bits(regions)
    c = skip.skip_corpus_load(_t(corpus))
    try:
        ix = skip.skip_ivfpq_build(c, _t(cent), _t(cb))
        ix.set_option(skip.SKIP_OPT_IVF_REFINE, refine)
        g_ids, g_sc = skip.skip_ivfpq_search_regions(ix, _t(regions), nprobe, k)
        q_ids, q_sc = skip.skip_ivfpq_search(ix, _t(regions), _t(offsets), nprobe, k, K)
        assert skip.skip_ivfpq_sync_status(ix) == skip.SKIP_OK
        off, ids, codes = (x.cpu().numpy() for x in skip.skip_ivfpq_lists(ix))
        ix.free()
        ix2 = skip.skip_ivfpq_load(_t(cent), _t(cb), _t(off), _t(ids, torch.int32), _t(codes))
        with pytest.raises(skip.SkipError) as e:
            ix2.set_option(skip.SKIP_OPT_IVF_REFINE, refine)
        assert e.value.status == skip.SKIP_EUNSUPPORTED
        ix2.free()
    finally:
        c.free()
    g_ids, g_sc, q_ids, q_sc = (x.cpu().numpy() for x in (g_ids, g_sc, q_ids, q_sc))
    lists, code_by_id = _lists_by_id(off, ids, codes, SPEC.N, cb.shape[0])
    gidx = {"offsets": off, "ids": ids.astype(np.int64), "codes": code_by_id, "lists": lists}
    # the oracle's shortlist one past ks (for the tie test) and its exact re-rank of all ks
    ext = 32
    s_ids, s_sc, _ = oracle.ivfpq_search(gidx, ce, cb.numpy(), qn, nprobe, ks + ext)
    o_ids, o_sc = oracle.ivfpq_search_refine(gidx, ce, cb.numpy(), qn, nprobe, ks, ks, cn)
    cs = np.sort(oracle.score_matrix(ce, qn), axis=1)[:, ::-1]
    truths = checker.region_truths(o_ids, o_sc, k)
    usable = []
    for r in range(qn.shape[0]):
        if cs[r, nprobe - 1] - cs[r, nprobe] <= PROBE_TIE:
            continue
        if s_ids[r, ks] >= 0 and s_sc[r, ks - 1] - s_sc[r, ks] <= PROBE_TIE:
            # A near tie in s^ at the shortlist's end only matters when one
            # of the tied entries could reach the exact top k.
            tied = np.nonzero((s_ids[r] >= 0) & (np.abs(s_sc[r] - s_sc[r, ks - 1]) <= PROBE_TIE))[0]
            if tied[-1] == ks + ext - 1:
                continue
            ex = oracle.scores_at(cn, qn, np.full(len(tied), r), s_ids[r, tied])
            if ex.max() >= truths[r].theta - checker.TAU:
                continue
        _, probs = checker.check_region(
            g_ids[r], g_sc[r], truths[r],
            extra_score=lambda i, r=r: float(oracle.scores_at(cn, qn, [r], [i])[0]))
        assert not probs, (r, probs[:3])
        usable.append(r)
    assert len(usable) >= qn.shape[0] // 2
    off_q = offsets.numpy()
    o_m_ids, o_m_sc = oracle.merge(o_ids, o_sc, k, off_q, K + 1)
    ok_r = set(usable)
    for q in range(off_q.shape[0] - 1):
        if not all(r in ok_r for r in range(off_q[q], off_q[q + 1])):
            continue

        def rescore(j, ids_, r0=off_q[q]):
            return oracle.scores_at(cn, qn, np.full(len(ids_), r0 + j), ids_)
        _, probs, _ = checker.check_question(q_ids[q], q_sc[q], o_m_ids[q], o_m_sc[q],
                                             truths[off_q[q]:off_q[q + 1]], K, g_ids[off_q[q]:off_q[q + 1]],
                                             rescore)
        assert not probs, (q, probs[:3])
