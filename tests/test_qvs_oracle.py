"""Pins of the QVS oracle (paper App. B.1 Def. B.1, Eq. qvs_score; Alg. 1
"QVS: prune") against values fixed outside the oracle: a hand-worked
example, the closed form with W_v = 0 and b_v = 0 (logit = <w_b, v>) against
a brute-force sort, a scaling invariant, and the count rule.
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
    fx = read_fixture("qvs_hand_example.txt")
    tok = _bits(fx["qvs_tokens"])[None]
    lg, idx, sc = oracle.qvs(tok, _bits(fx["fq"])[None], _bits(fx["wv"]), fx["bv"].astype(np.float32),
                             fx["wb"].astype(np.float32), fx["rho"])
    np.testing.assert_allclose(lg[0], fx["logits"], rtol=0, atol=1e-15)
    np.testing.assert_array_equal(idx[0], fx["kept"].astype(np.int32))
    np.testing.assert_allclose(sc[0], fx["scores"], rtol=1e-15, atol=0)


def test_zero_projection_ranks_by_content_bias():
    B, L, d = 3, 200, 64
    tokens, fq, wv, bv, wb = synth.make_qvs_inputs(B, L, d, seed=7)
    tokens[1, 50] = tokens[1, 10]  # an exact tie: index 10 ranks first
    zero_w = torch.zeros(d, d, dtype=torch.bfloat16)
    lg, idx, _ = oracle.qvs(synth.bf16_bits(tokens), synth.bf16_bits(fq), synth.bf16_bits(zero_w), None,
                            wb.numpy(), 0.3)
    want = tokens.double() @ wb.double()  # [B, L]
    np.testing.assert_allclose(lg, want.numpy(), rtol=0, atol=1e-12)
    n = oracle.qvs_count(L, 0.3)
    for b in range(B):
        order = np.lexsort((np.arange(L), -want[b].numpy()))
        np.testing.assert_array_equal(idx[b], order[:n])
    pos = list(idx[1])
    if 10 in pos and 50 in pos:
        assert pos.index(10) < pos.index(50)


def test_doubling_fq_and_wb_and_bv_doubles_the_logit():
    tokens, fq, wv, bv, wb = synth.make_qvs_inputs(2, 100, 32, seed=8)
    lg1, idx1, _ = oracle.qvs(synth.bf16_bits(tokens), synth.bf16_bits(fq), synth.bf16_bits(wv), bv.numpy(),
                              wb.numpy(), 0.4)
    lg2, idx2, _ = oracle.qvs(synth.bf16_bits(tokens), synth.bf16_bits(2 * fq), synth.bf16_bits(wv), bv.numpy(),
                              2 * wb.numpy(), 0.4)
    np.testing.assert_allclose(lg2, 2 * lg1, rtol=1e-12, atol=1e-14)
    np.testing.assert_array_equal(idx1, idx2)


@pytest.mark.parametrize("L,rho,want", [(576, 0.4, 231), (576, 0.11, 64), (576, 0.25, 144), (576, 0.9, 519),
                                        (10, 0.0, 0), (10, 1.0, 10), (7, 0.5, 4)])
def test_count_rule(L, rho, want):
    assert oracle.qvs_count(L, rho) == want
