"""Pins for the CPU oracle, each against something other than the oracle itself.

What is pinned and by what:

* the whole path (scores, per-region top-k, dedup by max, cut to K,
  padding, lower-id tie-break) -- a hand-worked integer example
  (tests/golden/hand_example.txt, paper §3.3 Eq. rcsr / App. B.2 Def. B.2);
* per-region top-k -- brute force by full sort on tiny inputs (numpy fp64
  product + lexsort, independent decode of bf16 bits);
* score indexing -- one-hot regions, for which s(r, i) = x_{i,t} and the
  top-k is the sorted column;
* score formula -- a region equal to a corpus row scores ||x||^2 against it
  and ranks it first among random unit rows;
* ranking direction -- planted nearest neighbours at known cosines;
* tie-break -- duplicated corpus rows;
* merge -- the invariants (unique ids, subset of the union, count
  min(K, |U|), non-increasing scores), monotonicity in the region set,
  the single-region and K <= k special cases, duplicated regions;
* e4m3 path -- the decode of all 256 codes against torch's float8_e4m3fn,
  brute force with row scales, and exact scaling by powers of two.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from tests._golden import read_fixture


def bf16_from_float(a):
    """Round-to-nearest-even fp32 -> bf16 bits via torch (input preparation)."""
    t = torch.as_tensor(np.asarray(a, dtype=np.float32)).to(torch.bfloat16)
    return synth.bf16_bits(t)


def decode_bf16(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def brute_topk(S, k):
    """Full sort of each row of S by (score desc, id asc)."""
    R, N = S.shape
    ids = np.empty((R, k), dtype=np.int64)
    sc = np.empty((R, k), dtype=np.float64)
    for r in range(R):
        order = np.lexsort((np.arange(N), -S[r]))[:k]
        ids[r] = order
        sc[r] = S[r, order]
    return ids, sc


# ---------------------------------------------------------------- golden

def test_hand_worked_example():
    fx = read_fixture("hand_example.txt")
    corpus = bf16_from_float(fx["corpus"])
    regions = bf16_from_float(fx["regions"])
    offsets = fx["offsets"].astype(np.int32)
    k, K = int(fx["k_region"]), int(fx["K"])
    reg_ids, reg_sc, out_ids, out_sc = oracle.retrieve(corpus, regions, offsets, k, K)
    np.testing.assert_array_equal(reg_ids, fx["region_ids"].astype(np.int64))
    np.testing.assert_array_equal(reg_sc, fx["region_scores"])
    np.testing.assert_array_equal(out_ids, fx["merged_ids"].astype(np.int64))
    np.testing.assert_array_equal(out_sc, fx["merged_scores"])


# ---------------------------------------------------------------- scores / top-k

@pytest.mark.parametrize("seed", [0, 1])
def test_region_topk_matches_full_sort(seed):
    rng = np.random.default_rng(seed)
    N, d, R, k = 3001, 64, 12, 9
    x = rng.standard_normal((N, d)).astype(np.float32)
    x /= np.linalg.norm(x, axis=1, keepdims=True)
    x[17] = x[5]            # duplicate rows: exact ties
    x[2900] = x[5]
    x[40] = 0.0             # a zero row scores exactly 0
    q = rng.standard_normal((R, d)).astype(np.float32)
    q /= np.linalg.norm(q, axis=1, keepdims=True)
    q[3] = x[5]             # ties at the top
    q[7] = q[6]             # duplicated region
    cb, qb = bf16_from_float(x), bf16_from_float(q)
    ids, sc = oracle.region_topk(cb, qb, k, nthreads=3)
    S = decode_bf16(qb) @ decode_bf16(cb).T
    bids, bsc = brute_topk(S, k)
    np.testing.assert_array_equal(ids, bids)
    np.testing.assert_array_equal(sc, bsc)
    assert list(ids[3][:3]) == [5, 17, 2900]


def test_score_matrix_is_the_inner_product():
    rng = np.random.default_rng(3)
    x = bf16_from_float(rng.standard_normal((50, 32)))
    q = bf16_from_float(rng.standard_normal((4, 32)))
    S = oracle.score_matrix(x, q)
    ref = decode_bf16(q) @ decode_bf16(x).T
    np.testing.assert_allclose(S, ref, rtol=0, atol=1e-12)


def test_one_hot_region_sorts_a_column():
    rng = np.random.default_rng(4)
    N, d, k = 2000, 48, 25
    cb = bf16_from_float(rng.standard_normal((N, d)))
    xs = decode_bf16(cb)
    for t in (0, 13, 47):
        e = np.zeros((1, d), dtype=np.float32)
        e[0, t] = 1.0
        ids, sc = oracle.region_topk(cb, bf16_from_float(e), k)
        order = np.lexsort((np.arange(N), -xs[:, t]))[:k]
        np.testing.assert_array_equal(ids[0], order)
        np.testing.assert_array_equal(sc[0], xs[order, t])


def test_self_score_is_squared_norm_and_ranks_first():
    cb = synth.bf16_bits(synth.random_bf16(4000, 256, seed=11))
    for j in (0, 1234, 3999):
        ids, sc = oracle.region_topk(cb, cb[j:j + 1], 1)
        xj = decode_bf16(cb[j])
        assert ids[0, 0] == j
        assert sc[0, 0] == float(np.sum(xj * xj))


def test_planted_nearest_neighbours():
    rng = np.random.default_rng(5)
    N, d, k = 5000, 256, 10
    x = rng.standard_normal((N, d))
    x /= np.linalg.norm(x, axis=1, keepdims=True)
    q = rng.standard_normal(d)
    q /= np.linalg.norm(q)
    planted = rng.choice(N, size=k, replace=False)
    for m, i in enumerate(planted):
        u = rng.standard_normal(d)
        u -= u.dot(q) * q
        u /= np.linalg.norm(u)
        c = 0.99 - 0.05 * m
        x[i] = c * q + math.sqrt(1 - c * c) * u
    ids, sc = oracle.region_topk(bf16_from_float(x), bf16_from_float(q[None]), k)
    np.testing.assert_array_equal(ids[0], planted)
    assert np.all(np.diff(sc[0]) < 0)
    assert abs(sc[0, 0] - 0.99) < 0.02


def test_duplicate_rows_lower_id_wins():
    cb = synth.bf16_bits(synth.random_bf16(300, 64, seed=2))
    cb[250] = cb[37]
    cb[299] = cb[37]
    q = cb[37:38]
    ids, _ = oracle.region_topk(cb, q, 1)
    assert ids[0, 0] == 37
    ids, sc = oracle.region_topk(cb, q, 3)
    assert list(ids[0]) == [37, 250, 299]
    assert sc[0, 0] == sc[0, 1] == sc[0, 2]


def test_k_beyond_N_pads():
    cb = synth.bf16_bits(synth.random_bf16(5, 16, seed=9))
    ids, sc = oracle.region_topk(cb, cb[:1], 8)
    assert sorted(ids[0, :5]) == [0, 1, 2, 3, 4]
    assert list(ids[0, 5:]) == [-1, -1, -1]
    assert np.all(np.isneginf(sc[0, 5:]))


# ---------------------------------------------------------------- merge

def _merge_inputs(seed, Q=6, k=7, N=800, d=32):
    rng = np.random.default_rng(seed)
    cb = bf16_from_float(rng.standard_normal((N, d)))
    counts = rng.integers(0, 6, size=Q)
    counts[0] = 1
    counts[1] = 0
    R = int(counts.sum())
    base = rng.standard_normal((Q, d))
    q = np.concatenate([base[i] + 0.3 * rng.standard_normal((c, d)) for i, c in enumerate(counts)])
    qb = bf16_from_float(q)
    offsets = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    return cb, qb, offsets, k


def _union_max(reg_ids, reg_sc, r0, r1):
    m = {}
    for r in range(r0, r1):
        for i, s in zip(reg_ids[r], reg_sc[r]):
            if i >= 0:
                m[int(i)] = max(m.get(int(i), -math.inf), float(s))
    return m


@pytest.mark.parametrize("K", [1, 5, 7, 12, 40])
def test_merge_invariants(K):
    cb, qb, offsets, k = _merge_inputs(10 + K)
    reg_ids, reg_sc, out_ids, out_sc = oracle.retrieve(cb, qb, offsets, k, K)
    for q in range(len(offsets) - 1):
        U = _union_max(reg_ids, reg_sc, offsets[q], offsets[q + 1])
        got = [(int(i), float(s)) for i, s in zip(out_ids[q], out_sc[q]) if i >= 0]
        n = min(K, len(U))
        assert len(got) == n
        assert len({i for i, _ in got}) == n                      # unique ids
        assert all(i in U and U[i] == s for i, s in got)           # max over regions
        assert len(U) <= k * (offsets[q + 1] - offsets[q])         # K' <= R k'
        assert all(a[1] >= b[1] for a, b in zip(got, got[1:]))     # non-increasing
        assert all(i == -1 for i in out_ids[q][n:])
        assert np.all(np.isneginf(out_sc[q][n:]))
        expect = sorted(U.items(), key=lambda t: (-t[1], t[0]))[:n]
        assert got == expect


def test_zero_region_question_is_all_padding():
    cb, qb, offsets, k = _merge_inputs(3)
    _, _, out_ids, out_sc = oracle.retrieve(cb, qb, offsets, k, 9)
    assert np.all(out_ids[1] == -1) and np.all(np.isneginf(out_sc[1]))


def test_merge_single_region_equals_region_list():
    cb, qb, _, k = _merge_inputs(4)
    offsets = np.arange(qb.shape[0] + 1, dtype=np.int32)
    reg_ids, reg_sc, out_ids, out_sc = oracle.retrieve(cb, qb, offsets, k, k)
    np.testing.assert_array_equal(out_ids, reg_ids)
    np.testing.assert_array_equal(out_sc, reg_sc)


def test_merge_with_K_at_most_k_is_global_top_of_max():
    cb, qb, offsets, k = _merge_inputs(5)
    K = 5
    _, _, out_ids, out_sc = oracle.retrieve(cb, qb, offsets, k, K)
    S = decode_bf16(qb) @ decode_bf16(cb).T
    for q in range(len(offsets) - 1):
        r0, r1 = offsets[q], offsets[q + 1]
        if r1 == r0:
            continue
        m = S[r0:r1].max(axis=0)
        order = np.lexsort((np.arange(m.size), -m))[:K]
        np.testing.assert_array_equal(out_ids[q], order)
        np.testing.assert_array_equal(out_sc[q], m[order])


def test_merge_monotone_in_regions_and_duplicate_regions_neutral():
    cb, qb, offsets, k = _merge_inputs(6)
    K = 15
    reg_ids, reg_sc = oracle.region_topk(cb, qb, k)
    a_ids, a_sc = oracle.merge(reg_ids, reg_sc, k, offsets, K)
    # Adding a region (its list appended) never lowers the merged score at any rank.
    extra_ids, extra_sc = oracle.region_topk(cb, qb[:1], k)
    for q in range(len(offsets) - 1):
        r0, r1 = offsets[q], offsets[q + 1]
        ids2 = np.concatenate([reg_ids[r0:r1], extra_ids])
        sc2 = np.concatenate([reg_sc[r0:r1], extra_sc])
        b_ids, b_sc = oracle.merge(ids2, sc2, k, np.array([0, r1 - r0 + 1], np.int32), K)
        assert np.all(b_sc[0] >= a_sc[q])
        # Duplicating every region leaves the output unchanged.
        ids3 = np.concatenate([reg_ids[r0:r1], reg_ids[r0:r1]])
        sc3 = np.concatenate([reg_sc[r0:r1], reg_sc[r0:r1]])
        c_ids, c_sc = oracle.merge(ids3, sc3, k, np.array([0, 2 * (r1 - r0)], np.int32), K)
        np.testing.assert_array_equal(c_ids[0], a_ids[q])
        np.testing.assert_array_equal(c_sc[0], a_sc[q])


# ---------------------------------------------------------------- e4m3

def test_e4m3_decode_matches_torch():
    codes = torch.arange(256, dtype=torch.int32).to(torch.uint8)
    ref = codes.view(torch.float8_e4m3fn).to(torch.float32).numpy().astype(np.float64)
    got = np.array([oracle.e4m3_value(b) for b in range(256)])
    nan = np.isnan(ref)
    assert np.array_equal(nan, np.isnan(got)) and nan.sum() == 2
    np.testing.assert_array_equal(got[~nan], ref[~nan])
    assert oracle.e4m3_value(0x01) == 2.0 ** -9     # smallest subnormal
    assert oracle.e4m3_value(0x7E) == 448.0         # largest finite


def test_bf16_decode():
    for h, v in ((0x3F80, 1.0), (0xBF80, -1.0), (0x0000, 0.0), (0x4049, 3.140625), (0x0001, 2.0 ** -133)):
        assert oracle.bf16_value(h) == v


def test_e4m3_brute_force_and_scale():
    spec = synth.WorkloadSpec("e4m3_small", 99, 1500, 64, "e4m3", 1, (6, 6), 8, 8, "gaussian")
    w = synth.make_workload(spec)
    cb = w.corpus.numpy()
    scale = w.row_scale.numpy()
    qb = synth.bf16_bits(w.regions)
    ids, sc = oracle.region_topk(cb, qb, 8, row_scale=scale)
    xs = torch.from_numpy(cb).view(torch.float8_e4m3fn).to(torch.float32).numpy().astype(np.float64)
    S = decode_bf16(qb) @ (xs * scale[:, None].astype(np.float64)).T
    bids, bsc = brute_topk(S, 8)
    np.testing.assert_array_equal(ids, bids)
    np.testing.assert_allclose(sc, bsc, rtol=0, atol=1e-12)
    # Scaling every row scale by 2^5 scales every score by exactly 2^5.
    _, sc2 = oracle.region_topk(cb, qb, 8, row_scale=scale * 32.0)
    np.testing.assert_array_equal(sc2, sc * 32.0)
    # An e4m3 corpus without scales is rejected.
    with pytest.raises(ValueError):
        oracle.region_topk(cb, qb, 8)


# ---------------------------------------------------------------- scores at chosen pairs

def test_scores_at_matches_numpy_product():
    """oracle.scores_at (the value the parity checker uses for ids outside
    the oracle's extended list) against a numpy fp64 product with an
    independent decode, at random (region, id) pairs of a bf16 and of an
    e4m3 corpus with per-row scales.  Region indices and ids are drawn
    independently, so a swapped index, a row taken from the wrong region or
    a missing scale changes the value; ids out of range give NaN."""
    rng = np.random.default_rng(7)
    N, d, R, n = 2000, 96, 9, 400
    x = rng.standard_normal((N, d)).astype(np.float32)
    q = rng.standard_normal((R, d)).astype(np.float32)
    cb, qb = bf16_from_float(x), bf16_from_float(q)
    reg = rng.integers(0, R, size=n)
    ids = rng.integers(0, N, size=n)
    got = oracle.scores_at(cb, qb, reg, ids)
    want = np.einsum("tj,tj->t", decode_bf16(qb)[reg], decode_bf16(cb)[ids])
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
    # e4m3 rows times their scales
    spec = synth.WorkloadSpec("e4m3_at", 98, N, d, "e4m3", 1, (R, R), 8, 8, "gaussian")
    w = synth.make_workload(spec)
    ce, sc = w.corpus.numpy(), w.row_scale.numpy()
    xs = torch.from_numpy(ce).view(torch.float8_e4m3fn).to(torch.float32).numpy().astype(np.float64)
    got = oracle.scores_at(ce, qb, reg, ids, row_scale=sc)
    want = np.einsum("tj,tj->t", decode_bf16(qb)[reg], xs[ids] * sc[ids, None].astype(np.float64))
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
    assert not np.allclose(got, np.einsum("tj,tj->t", decode_bf16(qb)[reg], xs[ids]))
    bad = oracle.scores_at(cb, qb, [0, 1], [-1, N])
    assert np.isnan(bad).all()
