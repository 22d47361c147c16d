"""Pins of the SKV gate oracle (paper App. B.4 Def. B.4, Eq. skv_score; the
Alg. 1 TopK after the SKV step) against values fixed outside the oracle:
a hand-worked example, torch's bf16 rounding, one-hot weights that read out
one input feature, the count rule, and properties of the selection.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from tests._golden import read_fixture


def _bits(x):
    return synth.bf16_bits(torch.as_tensor(np.asarray(x, np.float32)).to(torch.bfloat16))


def test_hand_example():
    fx = read_fixture("skv_hand_example.txt")
    d, H = int(fx["d"]), int(fx["H"])
    out = oracle.skv(_bits(fx["skv_corpus"]), fx["ids"].astype(np.int64), _bits(fx["qbar"]),
                     _bits(fx["vbar"]), _bits(fx["w1"]), fx["b1"].astype(np.float32),
                     fx["w2"].astype(np.float32), fx["b2"], tau=fx["tau"], rho=fx["rho"])
    assert fx["w1"].shape == (H, 5 * d)
    np.testing.assert_allclose(out["nu_all"], fx["nu_all"], rtol=1e-15, atol=0)
    np.testing.assert_array_equal(out["ids"], fx["out_ids"].astype(np.int64))
    np.testing.assert_allclose(out["nu"], fx["out_nu"], rtol=1e-15, atol=0)
    np.testing.assert_array_equal(out["count"], fx["count"].astype(np.int32))


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(3)
    # float32 values over many binades, including exact halfway cases and
    # values in the bf16 subnormal range.
    mant = rng.integers(0, 1 << 23, size=4000)
    expo = rng.integers(-140, 120, size=4000)
    vals = np.ldexp(1.0 + mant / float(1 << 23), expo) * rng.choice([-1.0, 1.0], size=4000)
    halves = np.ldexp(1.0 + (2 * rng.integers(0, 128, size=500) + 1) / 256.0, rng.integers(-20, 20, 500))
    vals = np.concatenate([vals, halves, [0.0, -0.0, 3.0e38, -3.0e38, 1e-40]]).astype(np.float32)
    want = torch.from_numpy(vals).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([oracle.bf16_round(float(v)) for v in vals], dtype=np.uint16)
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("block", range(5))
def test_one_hot_weights_read_each_feature(block):
    """W1 with +1 and -1 at one input column (units 0 and 1) and
    w2 = (1, -1) give logit = relu(f_t) - relu(-f_t) = f_t exactly, so nu
    reads out one feature: qbar, vbar, e, bf16(e*qbar), bf16(|e - qbar|)."""
    d, N, Q, K = 16, 40, 3, 6
    corpus = synth.random_bf16(N, d, seed=11)
    qbar = synth.random_bf16(Q, d, seed=12)
    vbar = synth.random_bf16(Q, d, seed=13)
    ids = synth.make_candidate_ids(N, Q, K, 1, seed=14)
    cf, qf, vf = corpus.float(), qbar.float(), vbar.float()
    for t in (0, 5, d - 1):
        col = block * d + t
        w1 = torch.zeros(2, 5 * d)
        w1[0, col], w1[1, col] = 1.0, -1.0
        out = oracle.skv(synth.bf16_bits(corpus), ids.numpy(), synth.bf16_bits(qbar), synth.bf16_bits(vbar),
                         synth.bf16_bits(w1.to(torch.bfloat16)), np.zeros(2, np.float32),
                         np.array([1.0, -1.0], np.float32), 0.0, tau=0.0, rho=1.0)
        for q in range(Q):
            for j in range(K):
                i = int(ids[q, j])
                if i < 0:
                    assert out["nu_all"][q, j] == -math.inf
                    continue
                e = cf[i]
                feat = [qf[q, t], vf[q, t], e[t],
                        (e[t] * qf[q, t]).to(torch.bfloat16).float(),
                        (e[t] - qf[q, t]).abs().to(torch.bfloat16).float()][block]
                want = 1.0 / (1.0 + math.exp(-float(feat)))
                assert out["nu_all"][q, j] == pytest.approx(want, rel=1e-14, abs=1e-300)


@pytest.mark.parametrize("n,rho,want", [(5, 0.6, 3), (4, 0.5, 2), (10, 0.3, 3), (0, 0.6, 0), (7, 1.0, 7),
                                        (3, 0.9, 3), (2000, 0.3, 600), (1, 0.3, 1), (8, 0.0, 0)])
def test_count_rule(n, rho, want):
    """ceil(rho |K|) (Alg. 1 TopK size) for two-decimal ratios."""
    assert oracle.skv_count(n, rho) == want


def _random_case(seed, N=300, d=32, Q=7, K=12, H=64):
    corpus = synth.random_bf16(N, d, seed=seed)
    qbar = synth.random_bf16(Q, d, seed=seed + 1)
    vbar = synth.random_bf16(Q, d, seed=seed + 2)
    empty = torch.tensor([0, 3, K, 1, 0, 5, 2])[:Q]
    ids = synth.make_candidate_ids(N, Q, K, empty, seed=seed + 3)
    w1, b1, w2, b2 = synth.make_skv_mlp(d, H, seed=seed + 4)
    return corpus, qbar, vbar, ids, w1, b1, w2, b2


def _run(case, tau, rho):
    corpus, qbar, vbar, ids, w1, b1, w2, b2 = case
    return oracle.skv(synth.bf16_bits(corpus), ids.numpy(), synth.bf16_bits(qbar), synth.bf16_bits(vbar),
                      synth.bf16_bits(w1), b1.numpy(), w2.numpy(), b2, tau=tau, rho=rho)


@pytest.mark.parametrize("tau,rho", [(0.5, 0.6), (0.0, 1.0), (0.7, 0.3), (0.5, 0.9)])
def test_selection_properties(tau, rho):
    case = _random_case(100)
    ids = case[3].numpy()
    out = _run(case, tau, rho)
    for q in range(ids.shape[0]):
        slots = [j for j in range(ids.shape[1]) if ids[q, j] >= 0]
        nu = out["nu_all"][q]
        gated = sorted(((nu[j], int(ids[q, j])) for j in slots if nu[j] >= tau), key=lambda x: (-x[0], x[1]))
        n = min(oracle.skv_count(len(slots), rho), len(gated))
        assert out["count"][q] == n
        assert list(out["ids"][q, :n]) == [g[1] for g in gated[:n]]
        assert np.all(out["ids"][q, n:] == -1) and np.all(np.isneginf(out["nu"][q, n:]))
        assert np.all(np.diff(out["nu"][q, :n]) <= 0)
        for j in range(ids.shape[1]):
            assert (nu[j] == -math.inf) == (ids[q, j] < 0)
    # tau 0 and rho 1 keep every candidate
    full = _run(case, 0.0, 1.0)
    assert list(full["count"]) == [int((ids[q] >= 0).sum()) for q in range(ids.shape[0])]


def test_raising_tau_never_adds():
    case = _random_case(200)
    prev = None
    for tau in (0.0, 0.3, 0.5, 0.6, 0.8, 1.0):
        out = _run(case, tau, 1.0)
        kept = [set(out["ids"][q, :out["count"][q]]) for q in range(out["ids"].shape[0])]
        if prev is not None:
            assert all(k <= p for k, p in zip(kept, prev))
        prev = kept


def test_fp32_evaluation_lands_within_bound():
    """An fp32 evaluation (numpy, its own summation order) of the same gate
    stays within the oracle's per-passage bound."""
    corpus, qbar, vbar, ids, w1, b1, w2, b2 = _random_case(300, d=64, H=128)
    out = _run((corpus, qbar, vbar, ids, w1, b1, w2, b2), 0.5, 0.6)
    d = corpus.shape[1]
    W = w1.float().numpy().astype(np.float32)
    C, Qb, Vb = corpus.float().numpy(), qbar.float().numpy(), vbar.float().numpy()
    for q in range(ids.shape[0]):
        c = (W[:, :d] @ Qb[q] + W[:, d:2 * d] @ Vb[q] + b1.numpy()).astype(np.float32)
        for j in range(ids.shape[1]):
            i = int(ids[q, j])
            if i < 0:
                continue
            e = C[i]
            eq = torch.from_numpy(e * Qb[q]).to(torch.bfloat16).float().numpy()
            ad = torch.from_numpy(np.abs(e - Qb[q])).to(torch.bfloat16).float().numpy()
            f = np.concatenate([e, eq, ad]).astype(np.float32)
            h = np.maximum(W[:, 2 * d:] @ f + c, np.float32(0))
            logit = np.float32(np.dot(w2.numpy(), h) + np.float32(b2))
            nu32 = np.float32(1) / (np.float32(1) + np.exp(-logit, dtype=np.float32))
            assert abs(float(nu32) - out["nu_all"][q, j]) <= out["bound"][q, j]
            assert 0 < out["bound"][q, j] < 2e-3
