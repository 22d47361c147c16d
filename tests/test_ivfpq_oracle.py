"""Pins of the IVF-PQ oracle (the index of §4.1 "Implementation" / App. I.4,
built and searched as in Jegou, Douze and Schmid, IEEE TPAMI 2011, with an
inner-product coarse quantizer) against values fixed outside the oracle: a
hand-worked example, brute force, and the closed form in which the index is
exact (every residual sub-vector a codeword, every list probed) and the
search must equal exact MIPS from the retrieval oracle.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests._golden import read_fixture


def _bits(x):
    return synth.bf16_bits(torch.as_tensor(np.asarray(x, np.float32)).to(torch.bfloat16))


def test_hand_example():
    fx = read_fixture("ivfpq_hand_example.txt")
    M, ksub, d = int(fx["M"]), int(fx["ksub"]), int(fx["d"])
    cb = fx["codebook"].astype(np.float32).reshape(M, ksub, d // M)
    corpus, cent, q = _bits(fx["ivf_corpus"]), _bits(fx["centroids"]), _bits(fx["queries"])
    idx = oracle.ivfpq_build(corpus, cent, cb)
    np.testing.assert_array_equal(idx["lists"], fx["lists"].astype(np.int32))
    np.testing.assert_array_equal(idx["codes"], fx["codes"].astype(np.uint8))
    for p, k, key in ((1, 2, "p1k2"), (1, 4, "p1k4"), (2, 3, "p2k3")):
        ids, sc, probes = oracle.ivfpq_search(idx, cent, cb, q, p, k)
        np.testing.assert_array_equal(ids, fx[key + "_ids"].astype(np.int64))
        np.testing.assert_array_equal(sc, fx[key + "_scores"])
        assert list(probes[0]) == [0, 1][:p]


def test_assign_and_encode_match_brute_force():
    rng = np.random.default_rng(5)
    N, d, C, M, ksub = 300, 32, 12, 8, 16
    corpus = synth.random_bf16(N, d, seed=1)
    cent = synth.random_bf16(C, d, seed=2)
    cent[7] = cent[3]  # duplicate centroid: rows assigned to 3, never 7
    cb = rng.normal(0, 0.05, size=(M, ksub, d // M)).astype(np.float32)
    cb[:, 9] = cb[:, 4]  # duplicate codeword: code 4, never 9
    lists = oracle.ivf_assign(synth.bf16_bits(corpus), synth.bf16_bits(cent))
    s = corpus.double() @ cent.double().T
    want = torch.argmax(s, dim=1).numpy()  # first maximum = lowest index
    np.testing.assert_array_equal(lists, want)
    assert not np.any(lists == 7)
    codes = oracle.pq_encode(synth.bf16_bits(corpus), synth.bf16_bits(cent), lists, cb)
    r = (corpus.double() - cent.double()[torch.as_tensor(lists, dtype=torch.long)]).numpy()
    for m in range(M):
        sub = r[:, m * (d // M):(m + 1) * (d // M)]
        dist = ((sub[:, None, :] - cb[m][None].astype(np.float64)) ** 2).sum(-1)
        np.testing.assert_array_equal(codes[:, m], np.argmin(dist, axis=1))
    assert not np.any(codes == 9)


def test_exact_index_equals_exact_mips():
    """Codebook = the residual sub-vectors themselves and nprobe = C: every
    code is exact, s^(q, i) = <q, x_i>, and the search is exact MIPS (the
    retrieval oracle's region_topk, a separate code path)."""
    spec = synth.WorkloadSpec("ivf_exact", 31, 256, 64, "bf16", 4, (2, 2), 12, 20, "clustered", 16)
    corpus, _, centres = synth.make_corpus(spec)
    cent = centres.to(torch.bfloat16)
    regions, _ = synth.make_regions(spec, centres)
    cb_bits = synth.bf16_bits(corpus)
    lists = oracle.ivf_assign(cb_bits, synth.bf16_bits(cent))
    M, ds = 16, 4
    r = (corpus.float() - cent.float()[torch.as_tensor(lists, dtype=torch.long)]).numpy()
    cb = np.stack([r[:, m * ds:(m + 1) * ds] for m in range(M)]).astype(np.float32)  # [M, 256, ds]
    idx = oracle.ivfpq_build(cb_bits, synth.bf16_bits(cent), cb)
    for m in range(M):  # every residual sub-vector is encoded exactly
        np.testing.assert_array_equal(cb[m][idx["codes"][:, m]], r[:, m * ds:(m + 1) * ds])
    q = synth.bf16_bits(regions)
    ids, sc, _ = oracle.ivfpq_search(idx, synth.bf16_bits(cent), cb, q, spec.centres, spec.k_region)
    e_ids, e_sc = oracle.region_topk(cb_bits, q, spec.k_region)
    np.testing.assert_allclose(sc, e_sc, rtol=0, atol=1e-12)
    for a, b, s in zip(ids, e_ids, e_sc):
        # ids agree except possibly inside exact score ties
        for t in range(len(a)):
            if a[t] != b[t]:
                assert np.isclose(s[t], s[min(t + 1, len(s) - 1)]) or np.isclose(s[t], s[max(t - 1, 0)])


def test_more_probes_never_lower_the_kth_score():
    spec = synth.WorkloadSpec("ivf_mono", 32, 3000, 64, "bf16", 4, (3, 3), 10, 20, "clustered", 32)
    corpus, _, centres = synth.make_corpus(spec)
    cent = synth.make_ivf_centroids(spec)
    cb = synth.make_pq_codebook(spec, 16).numpy()
    regions, _ = synth.make_regions(spec, centres)
    idx = oracle.ivfpq_build(synth.bf16_bits(corpus), synth.bf16_bits(cent), cb)
    q = synth.bf16_bits(regions)
    prev_sc, prev_probes = None, None
    for p in (1, 2, 4, 8, 16, 32):
        ids, sc, probes = oracle.ivfpq_search(idx, synth.bf16_bits(cent), cb, q, p, spec.k_region)
        if prev_sc is not None:
            assert np.all(sc[:, -1] >= prev_sc[:, -1])
            np.testing.assert_array_equal(probes[:, :prev_probes.shape[1]], prev_probes)
        prev_sc, prev_probes = sc, probes
        s_at = oracle.ivfpq_scores_at(idx, synth.bf16_bits(cent), cb, q, np.repeat(np.arange(q.shape[0]), spec.k_region),
                                      ids.ravel())
        np.testing.assert_allclose(s_at.reshape(ids.shape)[ids >= 0], sc[ids >= 0], rtol=0, atol=1e-12)
    # the index holds every id once
    assert sorted(idx["ids"].tolist()) == list(range(spec.N))
    assert idx["offsets"][-1] == spec.N


@pytest.mark.parametrize("nprobe,k", [(1, 5), (1, 30), (3, 12), (7, 40)])
def test_search_matches_brute_force_with_random_codes(nprobe, k):
    """An index given directly (random lists and random codes, so the build
    plays no part): for every region, the nprobe centroids with the largest
    <q, c_l> (lower l first on ties) are probed and every row of their lists
    is scored s^ = <q, c_list(i)> + sum_m <q_m, p_{m, code_{i,m}}> in fp64,
    then cut to the k best by (s^ desc, id asc), padded with (-1, -inf)."""
    rng = np.random.default_rng(17 + nprobe)
    N, d, C, M, ksub = 90, 32, 7, 8, 16
    ds = d // M
    cent = synth.random_bf16(C, d, seed=nprobe)
    cent[5] = cent[2]  # two equal centroid scores: the lower list is probed first
    q = synth.random_bf16(4, d, seed=10 + nprobe)
    cb = rng.normal(0, 0.1, size=(M, ksub, ds)).astype(np.float32)
    lists = rng.integers(0, C, N).astype(np.int32)
    codes = rng.integers(0, ksub, (N, M)).astype(np.uint8)
    order = np.argsort(lists, kind="stable")
    offsets = np.zeros(C + 1, np.int64)
    offsets[1:] = np.cumsum(np.bincount(lists, minlength=C))
    idx = {"lists": lists, "codes": codes, "offsets": offsets, "ids": order.astype(np.int64)}
    ids, sc, probes = oracle.ivfpq_search(idx, synth.bf16_bits(cent), cb, synth.bf16_bits(q), nprobe, k)
    qd, cd, cbd = q.double().numpy(), cent.double().numpy(), cb.astype(np.float64)
    for r in range(qd.shape[0]):
        cs = cd @ qd[r]
        want_probes = np.lexsort((np.arange(C), -cs))[:nprobe]
        np.testing.assert_array_equal(probes[r], want_probes)
        rows = np.nonzero(np.isin(lists, want_probes))[0]
        s = np.array([cs[lists[i]] + sum(qd[r, m * ds:(m + 1) * ds] @ cbd[m, codes[i, m]] for m in range(M))
                      for i in rows])
        top = np.lexsort((rows, -s))[:k]
        want_ids = np.full(k, -1, np.int64)
        want_sc = np.full(k, -np.inf)
        want_ids[:len(top)] = rows[top]
        want_sc[:len(top)] = s[top]
        np.testing.assert_array_equal(ids[r], want_ids)
        np.testing.assert_allclose(sc[r], want_sc, rtol=1e-12, atol=1e-12)


def test_refine_with_every_list_and_entry_is_exact_mips():
    """With every list probed and a shortlist as long as the corpus, the
    exact re-rank sees every row: the result is exact MIPS (region_topk, a
    separate code path), whatever the codebook.  With a shortlist of k the
    re-rank keeps the ids of the plain search and only re-scores them."""
    spec = synth.WorkloadSpec("ivf_refine", 33, 900, 64, "bf16", 4, (2, 2), 8, 16, "clustered", 16)
    corpus, _, centres = synth.make_corpus(spec)
    cent = synth.make_ivf_centroids(spec)
    cb = synth.make_pq_codebook(spec, 16).numpy()
    regions, _ = synth.make_regions(spec, centres)
    cbits, ce, q = synth.bf16_bits(corpus), synth.bf16_bits(cent), synth.bf16_bits(regions)
    idx = oracle.ivfpq_build(cbits, ce, cb)
    k = spec.k_region
    r_ids, r_sc = oracle.ivfpq_search_refine(idx, ce, cb, q, spec.centres, k, spec.N, cbits)
    e_ids, e_sc = oracle.region_topk(cbits, q, k)
    np.testing.assert_array_equal(r_ids, e_ids)
    np.testing.assert_allclose(r_sc, e_sc, rtol=0, atol=1e-12)
    p_ids, _, _ = oracle.ivfpq_search(idx, ce, cb, q, 4, k)
    s_ids, s_sc = oracle.ivfpq_search_refine(idx, ce, cb, q, 4, k, k, cbits)
    for a, b in zip(p_ids, s_ids):
        assert set(a.tolist()) == set(b.tolist())
    assert np.all(np.diff(s_sc, axis=1) <= 0)
