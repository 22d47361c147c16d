"""GPU parity of the SKV passage gate (App. B.4 Def. B.4, Eq. skv_score; the
Alg. 1 TopK after the SKV step) against the oracle (oracle/skv_oracle.c).

nu is compared slot by slot within the oracle's per-slot bound on an fp32
evaluation; the selection is compared exactly wherever the oracle's values
leave no doubt (no nu within twice the bound of tau, and the kept count's
cut clear of the next value), and otherwise checked to follow the rule on the
GPU's own nu.  Every input here comes from the seeded generators or from the
oracle; none from the CUDA path.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import paper_2607_25422_gb300 as skip
import synth
from tests._golden import read_fixture

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")


def _load(corpus):
    return skip.skip_corpus_load(corpus.to(DEV))


def _gate_gpu(c, ids, qbar, vbar, w1, b1, w2, b2, tau, rho):
    t = lambda x: x.to(DEV).contiguous()
    out = skip.skip_skv_gate(c, t(ids), t(qbar), t(vbar), t(w1), t(b1.float()), t(w2.float()), b2, tau, rho,
                             with_nu_all=True)
    assert skip.skip_sync_status(c) == skip.SKIP_OK
    return [x.cpu().numpy() for x in out]


def _gate_oracle(corpus, ids, qbar, vbar, w1, b1, w2, b2, tau, rho):
    b = synth.bf16_bits
    return oracle.skv(b(corpus), ids.numpy(), b(qbar), b(vbar), b(w1), b1.float().numpy(),
                      w2.float().numpy(), b2, tau=tau, rho=rho)


def check_gate(gpu, orc, ids, tau, rho):
    """gpu = (ids, nu, count, nu_all); orc = oracle.skv(...) on the same input."""
    g_ids, g_nu, g_cnt, g_all = gpu
    ids = np.asarray(ids)
    Q, K = ids.shape
    bound = orc["bound"]
    exact_q = 0
    strict_q = 0
    worst = 0.0
    for q in range(Q):
        for j in range(K):
            if ids[q, j] < 0:
                assert g_all[q, j] == -math.inf
            else:
                err = abs(float(g_all[q, j]) - orc["nu_all"][q, j])
                assert err <= bound[q, j], (q, j)
                worst = max(worst, err)
        # the rule applied to the GPU's own nu
        slots = [j for j in range(K) if ids[q, j] >= 0]
        gated = sorted(((float(g_all[q, j]), int(ids[q, j])) for j in slots if g_all[q, j] >= tau),
                       key=lambda x: (-x[0], x[1]))
        n = min(oracle.skv_count(len(slots), rho), len(gated))
        assert g_cnt[q] == n, q
        assert list(g_ids[q, :n]) == [x[1] for x in gated[:n]], q
        np.testing.assert_array_equal(g_nu[q, :n], np.array([x[0] for x in gated[:n]], np.float32))
        assert np.all(g_ids[q, n:] == -1) and np.all(np.isneginf(g_nu[q, n:]))
        # against the oracle where its values leave no doubt
        bq = 2 * max([bound[q, j] for j in slots], default=0.0)
        o_nu = sorted((orc["nu_all"][q, j] for j in slots), reverse=True)
        near_tau = any(abs(v - tau) <= bq for v in o_nu)
        on = int(orc["count"][q])
        o_g = [v for v in o_nu if v >= tau]
        cut_clear = on >= len(o_g) or on == 0 or (o_g[on - 1] - o_g[on] > bq)
        if not near_tau and cut_clear:
            assert g_cnt[q] == on, q
            assert set(g_ids[q, :on]) == set(orc["ids"][q, :on]), q
            exact_q += 1
        strict_q += int(g_cnt[q] == on and list(g_ids[q]) == list(orc["ids"][q]))
    print("largest |nu_gpu - nu_oracle| %.2e (bound median %.2e); %d of %d selections identical to the oracle's"
          % (worst, float(np.median(bound[ids >= 0])) if (ids >= 0).any() else 0.0, strict_q, Q))
    return exact_q


def test_hand_example_exact():
    """The hand-worked example, padded to d = 64 and H = 128 with zeros (the
    padding adds exact zeros to every sum)."""
    fx = read_fixture("skv_hand_example.txt")
    d0, H0, d, H = int(fx["d"]), int(fx["H"]), 64, 128
    corpus = torch.zeros(4, d)
    corpus[:, :d0] = torch.tensor(fx["skv_corpus"])
    qbar = torch.zeros(2, d)
    qbar[:, :d0] = torch.tensor(fx["qbar"])
    vbar = torch.zeros(2, d)
    vbar[:, :d0] = torch.tensor(fx["vbar"])
    w1 = torch.zeros(H, 5 * d)
    for blk in range(5):
        w1[:H0, blk * d:blk * d + d0] = torch.tensor(fx["w1"][:, blk * d0:(blk + 1) * d0])
    b1 = torch.zeros(H)
    b1[:H0] = torch.tensor(fx["b1"])
    w2 = torch.zeros(H)
    w2[:H0] = torch.tensor(fx["w2"])
    ids = torch.tensor(fx["ids"], dtype=torch.int64)
    bf = lambda x: x.to(torch.bfloat16)
    c = _load(bf(corpus))
    try:
        g_ids, g_nu, g_cnt, g_all = _gate_gpu(c, ids, bf(qbar), bf(vbar), bf(w1), b1, w2, float(fx["b2"]),
                                              float(fx["tau"]), float(fx["rho"]))
    finally:
        c.free()
    np.testing.assert_allclose(g_all, fx["nu_all"], rtol=0, atol=2e-7)
    np.testing.assert_array_equal(g_ids, fx["out_ids"].astype(np.int64))
    np.testing.assert_array_equal(g_cnt, fx["count"].astype(np.int32))
    np.testing.assert_allclose(g_nu, fx["out_nu"], rtol=0, atol=2e-7)


@pytest.mark.parametrize("block", range(5))
def test_one_hot_weights_read_each_feature(block):
    """One +1/-1 weight pair per hidden pair makes each logit one input
    feature exactly; this pins the feature blocks, their bf16 rounding and
    the column order of W1 on the tensor cores."""
    N, d, Q, K, H = 700, 128, 3, 40, 128
    corpus = synth.random_bf16(N, d, seed=21)
    qbar = synth.random_bf16(Q, d, seed=22)
    vbar = synth.random_bf16(Q, d, seed=23)
    ids = synth.make_candidate_ids(N, Q, K, torch.tensor([0, 7, 39]), seed=24)
    cols = [block * d + t for t in (0, 63, 64, d - 1)]
    c = _load(corpus)
    try:
        for col in cols:
            w1 = torch.zeros(H, 5 * d)
            w1[0, col], w1[1, col] = 1.0, -1.0
            w2 = torch.zeros(H)
            w2[0], w2[1] = 1.0, -1.0
            args = (ids, qbar, vbar, w1.to(torch.bfloat16), torch.zeros(H), w2, 0.0, 0.0, 1.0)
            g = _gate_gpu(c, *args)
            o = _gate_oracle(corpus, *args)
            ok = ids.numpy() >= 0
            np.testing.assert_allclose(g[3][ok], o["nu_all"][ok], rtol=0, atol=2e-7)
    finally:
        c.free()


CASES = [
    # N, d, Q, K, H, empty slots per question (cycled), tau, rho
    (5000, 768, 5, 50, 512, (0, 3, 50, 1, 10), 0.5, 0.6),
    (3000, 512, 9, 37, 256, (0, 1, 2), 0.5, 0.6),
    (4000, 1024, 3, 100, 128, (0, 40, 99), 0.6, 0.9),
    (2000, 64, 4, 1, 128, (0, 1), 0.5, 1.0),
    (3000, 256, 2, 2048, 384, (0, 1500), 0.4, 0.3),
    # enough slots that the MLP runs without the K split (one CTA pair per tile)
    (6000, 128, 64, 200, 512, (0, 7, 150), 0.5, 0.6),
    # one slot per question: more questions per tile than the MLP stages c_q for
    (3000, 128, 300, 1, 256, (0, 1), 0.5, 1.0),
    (20000, 64, 20000, 1, 512, (0, 1), 0.5, 1.0),
    # the largest K the selection ranks, and the smallest it sorts
    (3000, 128, 6, 256, 256, (0, 100, 255), 0.5, 0.6),
    (3000, 128, 5, 257, 256, (0, 1, 256), 0.5, 0.6),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "N%d_d%d_Q%d_K%d_H%d" % c[:5])
def test_random_gate(case):
    N, d, Q, K, H, empty, tau, rho = case
    corpus = synth.random_bf16(N, d, seed=N + d)
    qbar = synth.random_bf16(Q, d, seed=Q + 31)
    vbar = synth.random_bf16(Q, d, seed=Q + 32)
    emp = torch.tensor([empty[q % len(empty)] for q in range(Q)])
    ids = synth.make_candidate_ids(N, Q, K, emp, seed=K + 33)
    w1, b1, w2, b2 = synth.make_skv_mlp(d, H, seed=H + 34)
    args = (ids, qbar, vbar, w1, b1, w2, b2, tau, rho)
    c = _load(corpus)
    try:
        g = _gate_gpu(c, *args)
    finally:
        c.free()
    o = _gate_oracle(corpus, *args)
    exact = check_gate(g, o, ids, tau, rho)
    print("%s: %d of %d questions with an unambiguous selection, all equal to the oracle's" % (case[:5], exact, Q))


def test_full_size_gate_and_fused_path():
    """The clustered 1M workload: retrieval plus gate in one call equals the
    two calls in turn bit for bit; the gate on the oracle-independent
    synthetic candidate lists of the same shape (64 questions x 50, d = 768,
    H = 512) matches the oracle."""
    spec = synth.WORKLOADS["clustered_1m"]
    corpus, _, centres = synth.make_corpus(spec, device=DEV)
    regions, offsets = synth.make_regions(spec, centres, "cpu")
    qbar, vbar = synth.make_skv_queries(regions, offsets)
    w1, b1, w2, b2 = synth.make_skv_mlp(spec.d)
    t = lambda x: x.to(DEV).contiguous()
    c = skip.skip_corpus_load(corpus)
    try:
        reg, off = t(regions), t(offsets)
        m_ids, m_sc = skip.skip_retrieve(c, reg, off, spec.k_region, spec.K)
        sep = skip.skip_skv_gate(c, m_ids, t(qbar), t(vbar), t(w1), t(b1), t(w2), b2)
        fused = skip.skip_retrieve_skv(c, reg, off, spec.k_region, spec.K, t(qbar), t(vbar), t(w1), t(b1),
                                       t(w2), b2, with_merged=True)
        assert skip.skip_sync_status(c) == skip.SKIP_OK
        for a, b in zip(sep, fused[:3]):
            assert torch.equal(a, b)
        assert torch.equal(m_ids, fused[3]) and torch.equal(m_sc, fused[4])
        assert skip.skip_last_plan(c)["launches"] >= 5
        ids = synth.make_candidate_ids(spec.N, spec.Q, spec.K, torch.tensor([0, 0, 5, 20]).repeat(spec.Q // 4),
                                       seed=77)
        g = _gate_gpu(c, ids, qbar, vbar, w1, b1, w2, b2, 0.5, 0.6)
    finally:
        c.free()
    cn = synth.bf16_bits(corpus)
    del corpus
    torch.cuda.empty_cache()
    o = oracle.skv(cn, ids.numpy(), synth.bf16_bits(qbar), synth.bf16_bits(vbar), synth.bf16_bits(w1),
                   b1.numpy(), w2.numpy(), b2, tau=0.5, rho=0.6)
    exact = check_gate(g, o, ids, 0.5, 0.6)
    print("clustered_1m gate: %d of %d questions unambiguous and equal to the oracle's" % (exact, spec.Q))


def test_out_of_range_id_is_flagged_and_skipped():
    N, d, H = 500, 64, 128
    corpus = synth.random_bf16(N, d, seed=41)
    qbar = synth.random_bf16(1, d, seed=42)
    vbar = synth.random_bf16(1, d, seed=43)
    w1, b1, w2, b2 = synth.make_skv_mlp(d, H, seed=44)
    ids = torch.tensor([[3, N + 7, 9, -1]], dtype=torch.int64)
    t = lambda x: x.to(DEV).contiguous()
    c = _load(corpus)
    try:
        out = skip.skip_skv_gate(c, t(ids), t(qbar), t(vbar), t(w1), t(b1), t(w2), b2, 0.0, 1.0, with_nu_all=True)
        assert skip.skip_sync_status(c) == skip.SKIP_EINVAL
        nu_all = out[3].cpu().numpy()
        assert np.isneginf(nu_all[0, 1]) and np.isneginf(nu_all[0, 3])
        assert int(out[2][0]) == 2 and set(out[0][0, :2].tolist()) == {3, 9}
        assert skip.skip_sync_status(c) == skip.SKIP_OK
    finally:
        c.free()


def test_argument_errors():
    N, d, H = 300, 64, 128
    corpus = synth.random_bf16(N, d, seed=51)
    q = synth.random_bf16(2, d, seed=52).to(DEV)
    w1, b1, w2, b2 = synth.make_skv_mlp(d, H, seed=53)
    w1, b1, w2 = w1.to(DEV), b1.to(DEV), w2.to(DEV)
    ids = torch.zeros(2, 4, dtype=torch.int64, device=DEV)
    c = _load(corpus)
    try:
        with pytest.raises(skip.SkipError) as e:
            skip.skip_skv_gate(c, ids, q, q, w1[:100].contiguous(), b1[:100].contiguous(), w2[:100].contiguous(), b2)
        assert e.value.status == skip.SKIP_EINVAL
        with pytest.raises(skip.SkipError) as e:
            skip.skip_skv_gate(c, ids, q, q, w1, b1, w2, b2, rho_r=1.5)
        assert e.value.status == skip.SKIP_EINVAL
    finally:
        c.free()
    c = _load(synth.random_bf16(N, 48, seed=54))
    try:
        with pytest.raises(skip.SkipError) as e:
            skip.skip_skv_gate(c, ids, q[:, :48].contiguous(), q[:, :48].contiguous(), w1, b1, w2, b2)
        assert e.value.status == skip.SKIP_EUNSUPPORTED
    finally:
        c.free()
