"""GPU parity of QVS (paper App. B.1 Def. B.1, Eq. qvs_score; Alg. 1 "QVS:
prune") against the oracle (oracle/qvs_oracle.c).

Logits are compared token by token within TAU = 1e-4 (an fp32 evaluation of
two sums of at most 4,096 terms of unit-scale products: the probabilistic
bound lambda * sqrt(n) * 2^-24 * sum|terms| with lambda = 6 is below 2e-5
here); the kept set must hold every token whose oracle logit is more than
TAU above the n-th and otherwise only tokens within TAU of it; scores are
sigmoid of the GPU logits; kept rows are the tokens' bytes.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_25422_gb300 as skip
import synth
from tests._golden import read_fixture

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda")
TAU = 1e-4


def _run_gpu(tokens, fq, wv, bv, wb, rho, max_images=None, max_tokens=None):
    B, L, d = tokens.shape
    head = skip.skip_qvs_create(wv.to(DEV), None if bv is None else bv.to(DEV), wb.to(DEV),
                                max_images or max(B, 1), max_tokens or L)
    try:
        idx, score, kept, logits = skip.skip_qvs_prune(head, tokens.to(DEV), fq.to(DEV), rho, with_tokens=True,
                                                       with_logits=True)
        torch.cuda.synchronize()
        return idx.cpu().numpy(), score.cpu().numpy(), kept.cpu(), logits.cpu().numpy()
    finally:
        head.free()


def check(tokens, gpu, orc, rho):
    idx, score, kept, g_log = gpu
    o_log, o_idx, _ = orc
    B, L = o_log.shape
    n = oracle.qvs_count(L, rho)
    assert idx.shape == (B, n)
    np.testing.assert_allclose(g_log, o_log, rtol=0, atol=TAU)
    exact = 0
    for b in range(B):
        if n == 0:
            continue
        srt = np.sort(o_log[b])[::-1]
        theta = srt[n - 1]
        sure = set(np.nonzero(o_log[b] > theta + TAU)[0].tolist())
        band = set(np.nonzero(np.abs(o_log[b] - theta) <= TAU)[0].tolist())
        got = set(idx[b].tolist())
        assert len(got) == n and sure <= got and got - sure <= band, b
        # order: by the GPU's own logits, ties to the lower index
        order = sorted(idx[b].tolist(), key=lambda i: (-g_log[b, i], i))
        assert idx[b].tolist() == order, b
        np.testing.assert_allclose(score[b], 1 / (1 + np.exp(-g_log[b, idx[b]].astype(np.float64))), rtol=0,
                                   atol=1e-6)
        assert torch.equal(kept[b], tokens[b, torch.as_tensor(idx[b], dtype=torch.long)])
        exact += int(list(idx[b]) == list(o_idx[b]))
    return exact


def test_hand_example_exact():
    fx = read_fixture("qvs_hand_example.txt")
    d, dk = 8, int(fx["dk"])  # tokens padded from 2 to 8 values with zeros
    tok = torch.zeros(1, 6, d)
    tok[0, :, :2] = torch.tensor(fx["qvs_tokens"])
    wv = torch.zeros(dk, d)
    wv[:, :2] = torch.tensor(fx["wv"])
    wb = torch.zeros(d)
    wb[:2] = torch.tensor(fx["wb"])
    bf = lambda x: x.to(torch.bfloat16)
    idx, score, kept, logits = _run_gpu(bf(tok), bf(torch.tensor(fx["fq"]))[None], bf(wv),
                                        torch.tensor(fx["bv"], dtype=torch.float32), wb, float(fx["rho"]))
    np.testing.assert_array_equal(logits[0], fx["logits"].astype(np.float32))
    np.testing.assert_array_equal(idx[0], fx["kept"].astype(np.int32))
    np.testing.assert_allclose(score[0], fx["scores"], rtol=0, atol=1e-7)


CASES = [
    # B, L, d, dk, rho, with b_v
    (5, 576, 1024, 1024, 0.4, True),
    (3, 576, 256, 128, 0.11, False),
    (4, 100, 64, 256, 1.0, True),
    (2, 1, 64, 64, 0.4, True),
    (2, 4096, 128, 64, 0.25, True),
    (3, 300, 512, 512, 0.0, True),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "B%d_L%d_d%d_dk%d_rho%s" % c[:5])
def test_random(case):
    B, L, d, dk, rho, with_bv = case
    tokens, fq, wv, bv, wb = synth.make_qvs_inputs(B, L, d, seed=L + d)
    fq = fq[:, :dk].contiguous()
    wv = wv[:dk].contiguous()
    bv = bv[:dk].contiguous() if with_bv else None
    gpu = _run_gpu(tokens, fq, wv, bv, wb, rho)
    orc = oracle.qvs(synth.bf16_bits(tokens), synth.bf16_bits(fq), synth.bf16_bits(wv),
                     None if bv is None else bv.numpy(), wb.numpy(), rho)
    exact = check(tokens, gpu, orc, rho)
    print(case, "%d of %d kept lists identical to the oracle's" % (exact, B))


def test_full_size():
    """64 images x 576 tokens x 1024, d_k = 1024, rho_v = 0.4: the batch the
    benchmark times (bench.py --qvs), every image against the oracle."""
    B, L, d, rho = 64, 576, 1024, 0.4
    tokens, fq, wv, bv, wb = synth.make_qvs_inputs(B, L, d)
    gpu = _run_gpu(tokens, fq, wv, bv, wb, rho)
    orc = oracle.qvs(synth.bf16_bits(tokens), synth.bf16_bits(fq), synth.bf16_bits(wv), bv.numpy(), wb.numpy(),
                     rho)
    exact = check(tokens, gpu, orc, rho)
    print("full size: %d of %d kept lists identical to the oracle's" % (exact, B))


def test_argument_errors():
    tokens, fq, wv, bv, wb = synth.make_qvs_inputs(2, 50, 64, seed=3)
    head = skip.skip_qvs_create(wv.to(DEV), bv.to(DEV), wb.to(DEV), 2, 50)
    try:
        with pytest.raises(skip.SkipError) as e:
            skip.skip_qvs_prune(head, tokens.to(DEV), fq.to(DEV), 1.5)
        assert e.value.status == skip.SKIP_EINVAL
        big = torch.zeros(3, 50, 64, dtype=torch.bfloat16, device=DEV)
        with pytest.raises(skip.SkipError) as e:
            skip.skip_qvs_prune(head, big, torch.zeros(3, 64, dtype=torch.bfloat16, device=DEV), 0.4)
        assert e.value.status == skip.SKIP_EINVAL
    finally:
        head.free()
    with pytest.raises(skip.SkipError) as e:
        skip.skip_qvs_create(torch.zeros(64, 60, dtype=torch.bfloat16, device=DEV), None,
                             torch.zeros(60, device=DEV), 1, 10)
    assert e.value.status == skip.SKIP_EUNSUPPORTED
