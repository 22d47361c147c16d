"""Pins of the BSCA oracle (paper App. B.3 Def. B.3, Eq. bsca_edges and
bsca_attn) against values fixed outside the oracle: a hand-worked example,
dense attention (every edge kept) against torch's
scaled_dot_product_attention, single edges (out = W_V k_j), and the edge
count.
"""
import numpy as np
import torch

import oracle
import synth
from tests._golden import read_fixture


def _bits(x):
    return synth.bf16_bits(torch.as_tensor(np.asarray(x, np.float32)).to(torch.bfloat16))


def test_hand_example():
    fx = read_fixture("bsca_hand_example.txt")
    args = ([0, 3], [0, 2], _bits(fx["hv"]), _bits(fx["qh"]), _bits(fx["hk"]), _bits(fx["kh"]), _bits(fx["vh"]), 2)
    for dbar, key in ((1.0, "1"), (5.0 / 3.0, "2")):
        o = oracle.bsca(*args, dbar=dbar)
        assert o["tau"][0] == fx["tau" + key]
        np.testing.assert_array_equal(o["degree"], fx["deg" + key].astype(np.int32))
        np.testing.assert_allclose(o["out"], fx["out" + key], rtol=1e-15, atol=0)


def test_dense_equals_sdpa():
    x = synth.make_bsca_inputs(4, 30, 5, 12, 32, 16, 24, seed=3)
    b = synth.bf16_bits
    o = oracle.bsca(x["vis_offsets"], x["chunk_offsets"], b(x["hv"]), b(x["qh"]), b(x["hk"]), b(x["kh"]),
                    b(x["vh"]), 12, dbar=100.0)
    vo, co = x["vis_offsets"].tolist(), x["chunk_offsets"].tolist()
    for q in range(4):
        Q = x["qh"][vo[q]:vo[q + 1]].double()[None]
        K = x["kh"][co[q]:co[q + 1]].double()[None]
        V = x["vh"][co[q]:co[q + 1]].double()[None]
        want = torch.nn.functional.scaled_dot_product_attention(Q, K, V)[0].numpy()
        np.testing.assert_allclose(o["out"][vo[q]:vo[q + 1]], want, rtol=1e-12, atol=1e-12)
        assert np.all(o["degree"][vo[q]:vo[q + 1]] == co[q + 1] - co[q])


def test_edge_count_and_given_mask():
    x = synth.make_bsca_inputs(3, 40, 8, 16, 32, 16, 8, seed=4)
    b = synth.bf16_bits
    args = (x["vis_offsets"], x["chunk_offsets"], b(x["hv"]), b(x["qh"]), b(x["hk"]), b(x["kh"]), b(x["vh"]), 16)
    o = oracle.bsca(*args, dbar=4.0)
    vo = x["vis_offsets"].tolist()
    for q in range(3):
        assert o["degree"][vo[q]:vo[q + 1]].sum() == oracle.bsca_edges_count(40, 4.0)  # no ties in random data
    mask = (o["cos"] >= o["tau"][np.repeat(np.arange(3), 40)][:, None]).astype(np.uint8)
    co = x["chunk_offsets"].tolist()
    for q in range(3):
        mask[vo[q]:vo[q + 1], co[q + 1] - co[q]:] = 0
    o2 = oracle.bsca(*args, dbar=4.0, edge_mask=mask)
    np.testing.assert_array_equal(o2["out"], o["out"])
    # a token with exactly one edge gets W_V k_j
    one = np.nonzero(o["degree"] == 1)[0]
    for i in one[:5]:
        q = int(np.searchsorted(vo, i, side="right") - 1)
        j = int(np.nonzero(mask[i])[0][0])
        np.testing.assert_allclose(o["out"][i], x["vh"][co[q] + j].double().numpy(), rtol=0, atol=0)
