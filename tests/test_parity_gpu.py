"""GPU parity: the CUDA path against the oracle on small seeded inputs.

Sizes span several 256-row corpus tiles and 128-row query blocks with ragged
tails; both score kernels (tensor core and warp-dot) run every case that
they accept.  Per-region lists (skip_retrieve_regions) and merged lists
(skip_retrieve) are both checked; see tests/checker.py for the tolerance.
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

PATHS = {"tensor": skip.SKIP_PATH_TENSOR, "warp": skip.SKIP_PATH_WARP, "latency": skip.SKIP_PATH_LATENCY}


def _bits(t):
    return synth.bf16_bits(t)


def run_gpu(corpus, regions, offsets, k, K, path, scale=None, mma=0, options=()):
    dev = torch.device("cuda")
    c = skip.skip_corpus_load(corpus.to(dev), row_scale=None if scale is None else scale.to(dev))
    try:
        c.set_option(skip.SKIP_OPT_PATH, path)
        c.set_option(skip.SKIP_OPT_MMA, mma)
        for opt, val in options:
            c.set_option(opt, val)
        reg = regions.to(dev)
        rid, rsc = skip.skip_retrieve_regions(c, reg, k)
        oid, osc = skip.skip_retrieve(c, reg, torch.as_tensor(offsets).to(dev), k, K)
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        plan = skip.skip_last_plan(c)
        torch.cuda.synchronize()
        return rid.cpu().numpy(), rsc.cpu().numpy(), oid.cpu().numpy(), osc.cpu().numpy(), plan
    finally:
        c.free()


def oracle_truth(corpus_np, regions_np, offsets, k, K, scale_np=None, extra=64):
    """The oracle's extended per-region lists and its merged lists with one
    slot past K (for the merged K / K+1 gap)."""
    N = corpus_np.shape[0]
    kk = min(N, k + extra)
    ids_ext, sc_ext = oracle.region_topk(corpus_np, regions_np, kk, row_scale=scale_np)
    oid, osc = oracle.merge(ids_ext, sc_ext, k, np.asarray(offsets, np.int32), K + 1)
    return ids_ext, sc_ext, oid, osc


def assert_parity(corpus_np, regions_np, offsets, k, K, gpu, truth, scale_np=None):
    rid, rsc, oid, osc, plan = gpu
    ids_ext, sc_ext, o_ids, o_sc = truth
    truths = checker.region_truths(ids_ext, sc_ext, k)
    extra = lambda r: (lambda i: float(oracle.scores_at(corpus_np, regions_np, [r], [i], row_scale=scale_np)[0]))
    bad = []
    n_exact = 0
    for r, t in enumerate(truths):
        ex, probs = checker.check_region(rid[r], rsc[r], t, extra_score=extra(r))
        n_exact += ex
        if probs:
            bad.append(("region", r, probs[:3]))
    q_exact = 0
    for q in range(len(offsets) - 1):
        r0, r1 = offsets[q], offsets[q + 1]
        ts = truths[r0:r1]
        rescore = checker.exact_rescore(corpus_np, regions_np[r0:r1], ts, row_scale=scale_np)
        ex, probs, _ = checker.check_question(oid[q], osc[q], o_ids[q], o_sc[q], ts, K, rid[r0:r1], rescore)
        q_exact += ex
        if probs:
            bad.append(("question", q, probs[:3]))
    assert not bad, "plan %s: %s" % (plan, bad[:5])
    return n_exact, q_exact


def ragged_offsets(Q, R, seed):
    rng = np.random.default_rng(seed)
    cuts = np.sort(rng.integers(0, R + 1, size=Q - 1))
    return np.concatenate([[0], cuts, [R]]).astype(np.int32)


@pytest.mark.parametrize("path", ["tensor", "warp"])
def test_hand_example_exact(path):
    fx = read_fixture("hand_example.txt")
    # d must be a multiple of 16: pad the 4 coordinates with zeros.
    corpus = np.zeros((8, 16), np.float32)
    corpus[:, :4] = fx["corpus"]
    regions = np.zeros((4, 16), np.float32)
    regions[:, :4] = fx["regions"]
    ct = torch.from_numpy(corpus).to(torch.bfloat16)
    rt = torch.from_numpy(regions).to(torch.bfloat16)
    offsets = fx["offsets"].astype(np.int32)
    rid, rsc, oid, osc, plan = run_gpu(ct, rt, offsets, 3, 4, PATHS[path])
    assert plan["path"] == ("tensor" if path == "tensor" else "warpdot")
    np.testing.assert_array_equal(rid, fx["region_ids"].astype(np.int64))
    np.testing.assert_array_equal(rsc, fx["region_scores"].astype(np.float32))
    np.testing.assert_array_equal(oid, fx["merged_ids"].astype(np.int64))
    np.testing.assert_array_equal(osc, fx["merged_scores"].astype(np.float32))


CASES = [
    # N, d, R, Q, k, K
    (3000, 64, 1, 1, 5, 5),
    (3001, 128, 7, 3, 13, 20),
    (5000, 768, 33, 5, 10, 20),
    (2600, 256, 130, 17, 64, 100),
    (300, 64, 5, 2, 300, 40),
    (20000, 512, 257, 40, 100, 100),
    (70000, 768, 64, 8, 20, 50),
]


@pytest.mark.parametrize("path", ["tensor", "warp"])
@pytest.mark.parametrize("case", CASES, ids=lambda c: "N%d_d%d_R%d_k%d_K%d" % (c[0], c[1], c[2], c[4], c[5]))
def test_random_bf16(case, path):
    N, d, R, Q, k, K = case
    if path == "warp" and R > 64:
        pytest.skip("warp-dot path re-reads the corpus per 8 regions; covered at R <= 64")
    ct = synth.random_bf16(N, d, seed=N + d)
    rt = synth.random_bf16(R, d, seed=R + 7)
    offsets = ragged_offsets(Q, R, seed=N)
    cn, rn = _bits(ct), _bits(rt)
    truth = oracle_truth(cn, rn, offsets, k, K)
    gpu = run_gpu(ct, rt, offsets, k, K, PATHS[path])
    assert_parity(cn, rn, offsets, k, K, gpu, truth)


def test_single_cta_mma():
    """The single-CTA (cta_group::1) tensor path over several query blocks,
    the last one partial, and a ragged corpus tail; launched without
    thread-block clusters."""
    N, d, R, Q, k, K = 40000, 256, 700, 30, 16, 40
    ct = synth.random_bf16(N, d, seed=77)
    rt = synth.random_bf16(R, d, seed=78)
    offsets = ragged_offsets(Q, R, seed=79)
    cn, rn = _bits(ct), _bits(rt)
    truth = oracle_truth(cn, rn, offsets, k, K)
    gpu = run_gpu(ct, rt, offsets, k, K, skip.SKIP_PATH_TENSOR, mma=1)
    assert gpu[4]["cluster"] == 1 and gpu[4]["mma"] == "single"
    assert_parity(cn, rn, offsets, k, K, gpu, truth)


PAIR_CASES = [
    # N, d, R, Q, k, K: R spans 1..5 query blocks (odd counts leave a padded CTA)
    (9000, 128, 100, 6, 10, 20),
    (33333, 256, 300, 20, 16, 40),
    (20000, 768, 512, 32, 20, 50),
    (12000, 512, 620, 40, 100, 100),
]


@pytest.mark.parametrize("case", PAIR_CASES, ids=lambda c: "N%d_d%d_R%d_k%d" % (c[0], c[1], c[2], c[4]))
def test_pair_mma(case):
    """The CTA-pair (cta_group::2) tensor path, forced even for one block."""
    N, d, R, Q, k, K = case
    ct = synth.random_bf16(N, d, seed=N + 5)
    rt = synth.random_bf16(R, d, seed=R + 11)
    offsets = ragged_offsets(Q, R, seed=R)
    cn, rn = _bits(ct), _bits(rt)
    truth = oracle_truth(cn, rn, offsets, k, K)
    gpu = run_gpu(ct, rt, offsets, k, K, skip.SKIP_PATH_TENSOR, mma=2)
    assert gpu[4]["mma"] == "pair" and gpu[4]["cluster"] == 2
    assert_parity(cn, rn, offsets, k, K, gpu, truth)


BOUND_CASES = [
    # N, d, R, Q, k, K, mma, resident option (0 auto, 2 forced), resident expected
    (70000, 768, 512, 32, 20, 50, 2, 0, 0),
    (45000, 256, 300, 20, 100, 100, 2, 0, 0),
    # forced: sets in global memory that fill (rescans from L2) and grow
    # past 32 keys (sorted in place at the end of an item)
    (45000, 256, 300, 20, 100, 100, 2, 2, 1),
    (30000, 128, 200, 10, 7, 16, 1, 0, 0),
    # 33 sample tiles in 8 chunks, k = 16: four-slot lists kept in registers
    (400000, 128, 256, 16, 16, 40, 2, 0, 0),
    # k = 4: items of 97 tiles leave about 16 keys per set, so the query
    # blocks stay resident by default
    (300000, 128, 300, 20, 4, 16, 2, 0, 1),
    # d = 512, k = 100 with a four-key bounding pass over 50 sample chunks,
    # forced resident
    (700000, 512, 300, 20, 100, 100, 2, 2, 1),
]


@pytest.mark.parametrize("case", BOUND_CASES,
                         ids=lambda c: "N%d_d%d_R%d_k%d_mma%d_res%d" % (c[0], c[1], c[2], c[4], c[6], c[7]))
def test_bounding_pass(case):
    """The bounding pass (every 48th corpus tile first, its merged top-k
    seeding each row's shared threshold) forced on, with the query blocks
    resident where the case expects it: the oracle's results, and exactly
    the same keys as without the bounding pass (sets in shared memory)."""
    N, d, R, Q, k, K, mma, res_opt, res_expected = case
    ct = synth.random_bf16(N, d, seed=N + 7)
    rt = synth.random_bf16(R, d, seed=R + 13)
    offsets = ragged_offsets(Q, R, seed=R + 1)
    cn, rn = _bits(ct), _bits(rt)
    truth = oracle_truth(cn, rn, offsets, k, K)
    on = run_gpu(ct, rt, offsets, k, K, skip.SKIP_PATH_TENSOR, mma=mma,
                 options=((skip.SKIP_OPT_BOUND, 2), (skip.SKIP_OPT_RESIDENT, res_opt)))
    off = run_gpu(ct, rt, offsets, k, K, skip.SKIP_PATH_TENSOR, mma=mma, options=((skip.SKIP_OPT_BOUND, 1),))
    assert on[4]["bound"] == 1 and off[4]["bound"] == 0
    assert on[4]["resident_queries"] == res_expected and off[4]["resident_queries"] == 0
    assert_parity(cn, rn, offsets, k, K, on, truth)
    for a, b in zip(on[:4], off[:4]):
        np.testing.assert_array_equal(a, b)


def test_clustered_near_ties():
    """Clustered rows put many candidates within 2e-3 of the k-th score."""
    spec = synth.WorkloadSpec("clustered_small", 11, 60000, 256, "bf16", 12, (1, 12), 20, 50, "clustered", 64)
    w = synth.make_workload(spec)
    cn, rn = _bits(w.corpus), _bits(w.regions)
    offsets = w.offsets.numpy()
    truth = oracle_truth(cn, rn, offsets, spec.k_region, spec.K, extra=400)
    gpu = run_gpu(w.corpus, w.regions, offsets, spec.k_region, spec.K, skip.SKIP_PATH_TENSOR)
    assert_parity(cn, rn, offsets, spec.k_region, spec.K, gpu, truth)


@pytest.mark.parametrize("path", ["tensor", "warp", "latency"])
def test_duplicate_rows_and_ties(path):
    ct = synth.random_bf16(4000, 128, seed=5)
    ct[1000] = ct[17]
    ct[3999] = ct[17]
    ct[2500] = ct[17]
    ct[100] = 0
    ct[101] = 0
    rt = torch.stack([ct[17], ct[17], ct[2500], torch.zeros_like(ct[0]), ct[5]]).clone()
    rt[3, 0] = 1.0  # scores x_{i,0}: many exact ties among rows
    offsets = np.array([0, 2, 2, 5], np.int32)  # a question with no regions
    k, K = 6, 9
    cn, rn = _bits(ct), _bits(rt)
    truth = oracle_truth(cn, rn, offsets, k, K)
    rid, rsc, oid, osc, plan = run_gpu(ct, rt, offsets, k, K, PATHS[path])
    assert list(rid[0][:4]) == [17, 1000, 2500, 3999]
    np.testing.assert_array_equal(rid[:3], truth[0][:3, :k])
    assert np.all(oid[1] == -1) and np.all(np.isneginf(osc[1]))
    assert_parity(cn, rn, offsets, k, K, (rid, rsc, oid, osc, plan), truth)


@pytest.mark.parametrize("case", [(5000, 1024, 3, 1, 10, 100), (4000, 128, 12, 4, 7, 30),
                                  (2999, 64, 1, 1, 40, 40)])
def test_random_e4m3(case):
    N, d, R, Q, k, K = case
    spec = synth.WorkloadSpec("e4m3_case", 20 + R, N, d, "e4m3", Q, (R // Q, R // Q), k, K, "gaussian")
    corpus, scale, _ = synth.make_corpus(spec)
    rt = synth.random_bf16(R, d, seed=R + 3)
    offsets = ragged_offsets(Q, R, seed=d)
    cn, rn, sn = corpus.numpy(), _bits(rt), scale.numpy()
    truth = oracle_truth(cn, rn, offsets, k, K, scale_np=sn)
    gpu = run_gpu(corpus, rt, offsets, k, K, skip.SKIP_PATH_AUTO, scale=scale)
    assert_parity(cn, rn, offsets, k, K, gpu, truth, scale_np=sn)


@pytest.mark.parametrize("case", [(5000, 1024, 32, 1, 10, 100), (7001, 80, 20, 4, 7, 30),
                                  (3000, 256, 130, 9, 16, 40), (20000, 512, 40, 5, 50, 60)],
                         ids=lambda c: "N%d_d%d_R%d_k%d" % (c[0], c[1], c[2], c[4]))
def test_e4m3_tensor_path(case):
    """e4m3 corpus on the tensor cores (tiles widened to bf16 in shared
    memory, row scales applied to the accumulator)."""
    N, d, R, Q, k, K = case
    spec = synth.WorkloadSpec("e4m3_tc", 60 + d, N, d, "e4m3", Q, (1, 1), k, K, "gaussian")
    corpus, scale, _ = synth.make_corpus(spec)
    rt = synth.random_bf16(R, d, seed=R + 5)
    offsets = ragged_offsets(Q, R, seed=N)
    cn, rn, sn = corpus.numpy(), _bits(rt), scale.numpy()
    truth = oracle_truth(cn, rn, offsets, k, K, scale_np=sn)
    gpu = run_gpu(corpus, rt, offsets, k, K, skip.SKIP_PATH_TENSOR, scale=scale)
    assert gpu[4]["path"] == "tensor"
    assert_parity(cn, rn, offsets, k, K, gpu, truth, scale_np=sn)


LATENCY_CASES = [
    # dtype, N, d, R, Q, k, K
    ("bf16", 10000, 64, 1, 1, 5, 5),
    ("bf16", 30001, 768, 32, 4, 10, 20),
    ("bf16", 5000, 256, 7, 3, 50, 60),
    ("bf16", 2000, 128, 20, 5, 64, 80),
    # register-set widths 4, 8, 12 and 16 at their upper ends
    ("bf16", 50000, 512, 24, 6, 3, 8),
    ("bf16", 3000, 64, 9, 3, 8, 16),
    ("bf16", 20000, 128, 16, 4, 12, 24),
    ("bf16", 40003, 256, 32, 8, 16, 30),
    ("e4m3", 6000, 1024, 32, 1, 10, 100),
    ("e4m3", 7001, 80, 5, 2, 7, 20),
    ("e4m3", 20000, 512, 17, 3, 30, 40),
]


@pytest.mark.parametrize("case", LATENCY_CASES, ids=lambda c: "%s_N%d_d%d_R%d_k%d" % (c[0], c[1], c[2], c[3], c[5]))
def test_small_batch_tensor_path(case):
    """Small region batches with the corpus tile as the streamed MMA operand
    (bf16, or e4m3 with the queries split into three e4m3 parts)."""
    dt, N, d, R, Q, k, K = case
    if dt == "bf16":
        corpus, scale = synth.random_bf16(N, d, seed=N + 1), None
        cn, sn = _bits(corpus), None
    else:
        spec = synth.WorkloadSpec("lat_e4m3", 80 + R, N, d, "e4m3", Q, (1, 1), k, K, "gaussian")
        corpus, scale, _ = synth.make_corpus(spec)
        cn, sn = corpus.numpy(), scale.numpy()
    rt = synth.random_bf16(R, d, seed=R + 13)
    offsets = ragged_offsets(Q, R, seed=N + R)
    rn = _bits(rt)
    truth = oracle_truth(cn, rn, offsets, k, K, scale_np=sn)
    gpu = run_gpu(corpus, rt, offsets, k, K, skip.SKIP_PATH_LATENCY, scale=scale)
    assert gpu[4]["path"] == "latency"
    assert_parity(cn, rn, offsets, k, K, gpu, truth, scale_np=sn)


def test_host_entry_point_matches_device():
    ct = synth.random_bf16(9000, 256, seed=8)
    rt = synth.random_bf16(40, 256, seed=9)
    offsets = ragged_offsets(6, 40, seed=3)
    dev = torch.device("cuda")
    c = skip.skip_corpus_load(ct.to(dev))
    try:
        a_ids, a_sc = skip.skip_retrieve(c, rt.to(dev), torch.as_tensor(offsets).to(dev), 12, 30)
        b_ids, b_sc = skip.skip_retrieve_host(c, rt.pin_memory(), torch.as_tensor(offsets), 12, 30)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(a_ids.cpu().numpy(), b_ids.numpy())
        np.testing.assert_array_equal(a_sc.cpu().numpy(), b_sc.numpy())
    finally:
        c.free()


def test_argument_errors():
    dev = torch.device("cuda")
    ct = synth.random_bf16(100, 32, seed=1).to(dev)
    c = skip.skip_corpus_load(ct)
    try:
        rt = ct[:4]
        off = torch.tensor([0, 4], dtype=torch.int32, device=dev)
        for bad in (dict(k_region=0, K=5), dict(k_region=101, K=5), dict(k_region=5, K=0),
                    dict(k_region=2000, K=5)):
            with pytest.raises(skip.SkipError) as e:
                skip.skip_retrieve(c, rt, off, **bad)
            assert e.value.status == skip.SKIP_EINVAL
        with pytest.raises(skip.SkipError):
            skip.skip_corpus_load(torch.zeros(10, 24, dtype=torch.bfloat16, device=dev))
        with pytest.raises(skip.SkipError):
            skip.skip_corpus_set_option(c, skip.SKIP_OPT_PATH, 7)
    finally:
        c.free()
