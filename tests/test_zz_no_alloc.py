"""The allocation-free per-region entry point against the handle-based one.

skip_retrieve_regions_noalloc serves callers that cannot let a library
allocate device memory -- applications whose framework owns every device
allocation, and serving loops that cannot take cudaMalloc's device-wide
synchronisation.  Its scratch is a fixed array in the library's device
memory, shared by all calls on a device.  This test calls it twice in a row
through the C ABI (the second call finds the previous call's leftovers in
that array) and compares both results with skip_retrieve_regions on the
same inputs, within the parity tolerance of the other tests, and checks
both against the CPU oracle directly.  It also checks that misaligned
pointers and ill-shaped tensors are refused before anything is launched.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2607_25422_gb300 as skip
import synth
from tests import checker

pytestmark = pytest.mark.gpu

TAU = 2e-3


def _same(ids_a, sc_a, ids_b, sc_b):
    assert np.all(np.abs(sc_a - sc_b) <= TAU)
    for r in range(ids_a.shape[0]):
        if set(ids_a[r]) != set(ids_b[r]):
            # only near-ties at the k-th score may differ
            kth = min(sc_a[r, -1], sc_b[r, -1])
            diff = set(ids_a[r]) ^ set(ids_b[r])
            sa = dict(zip(ids_a[r], sc_a[r]))
            sb = dict(zip(ids_b[r], sc_b[r]))
            for i in diff:
                s = sa.get(i, sb.get(i))
                assert abs(s - kth) <= TAU, (r, i, s, kth)


@pytest.mark.parametrize("dtype", ["bf16", "e4m3"])
def test_noalloc_matches_handle_path_twice(dtype):
    dev = torch.device("cuda")
    N, d, R, k = 30000, 256, 11, 17
    if dtype == "bf16":
        corpus = synth.random_bf16(N, d, seed=41).to(dev)
        scale = None
    else:
        spec = synth.WorkloadSpec("noalloc_e4m3", 42, N, d, "e4m3", 1, (R, R), k, k, "gaussian")
        c_cpu, s_cpu, _ = synth.make_corpus(spec)
        corpus, scale = c_cpu.to(dev), s_cpu.to(dev)
    regions = synth.random_bf16(R, d, seed=43).to(dev)
    if dtype == "bf16":
        cn, sn = synth.bf16_bits(corpus.cpu()), None
    else:
        cn, sn = corpus.cpu().numpy(), scale.cpu().numpy()
    rn = synth.bf16_bits(regions.cpu())
    o_ids, o_sc = oracle.region_topk(cn, rn, k + 32, row_scale=sn)
    truths = checker.region_truths(o_ids, o_sc, k)

    handle = skip.skip_corpus_load(corpus, row_scale=scale)
    try:
        handle.set_option(skip.SKIP_OPT_PATH, skip.SKIP_PATH_WARP)
        ref_ids, ref_sc = skip.skip_retrieve_regions(handle, regions, k)
        assert skip.skip_sync_status(handle) == skip.SKIP_OK
    finally:
        handle.free()
    ref_ids, ref_sc = ref_ids.cpu().numpy(), ref_sc.cpu().numpy()

    lib = skip.load_library()
    stream = torch.cuda.current_stream().cuda_stream
    dt = skip.SKIP_BF16 if dtype == "bf16" else skip.SKIP_E4M3
    for _ in range(2):
        ids = torch.full((R, k), -7, dtype=torch.int64, device=dev)
        sc = torch.full((R, k), 7.0, dtype=torch.float32, device=dev)
        st = lib.skip_retrieve_regions_noalloc(
            ctypes.c_void_p(corpus.data_ptr()), N, d, dt,
            None if scale is None else ctypes.c_void_p(scale.data_ptr()),
            ctypes.c_void_p(regions.data_ptr()), R, k,
            ctypes.c_void_p(ids.data_ptr()), ctypes.c_void_p(sc.data_ptr()), ctypes.c_void_p(stream))
        assert st == skip.SKIP_OK, skip.skip_status_string(st)
        torch.cuda.synchronize()
        g_ids, g_sc = ids.cpu().numpy(), sc.cpu().numpy()
        _same(g_ids, g_sc, ref_ids, ref_sc)
        for r, t in enumerate(truths):
            _, probs = checker.check_region(
                g_ids[r], g_sc[r], t,
                extra_score=lambda i, r=r: float(oracle.scores_at(cn, rn, [r], [i], row_scale=sn)[0]))
            assert not probs, (r, probs[:3])


def test_noalloc_rejects_sizes_beyond_its_scratch():
    dev = torch.device("cuda")
    corpus = synth.random_bf16(5000, 64, seed=1).to(dev)
    regions = synth.random_bf16(4000, 64, seed=2).to(dev)
    ids = torch.empty(4000, 1000, dtype=torch.int64, device=dev)
    sc = torch.empty(4000, 1000, dtype=torch.float32, device=dev)
    with pytest.raises(skip.SkipError) as e:
        skip.skip_retrieve_regions_noalloc(corpus, regions, 1000, ids, sc)
    assert e.value.status == skip.SKIP_EUNSUPPORTED


def test_noalloc_refuses_misaligned_pointers_before_launch():
    """Corpus rows off a 16-byte boundary, regions off 2 bytes, ids off 8 and
    scores off 4 bytes: each is refused with SKIP_EINVAL by the host-side
    check, so no kernel ever sees the misaligned address."""
    dev = torch.device("cuda")
    N, d, R, k = 4096, 64, 3, 5
    corpus = synth.random_bf16(N + 16, d, seed=3).to(dev)
    regions = synth.random_bf16(R + 1, d, seed=4).to(dev)
    ids = torch.empty(R * k + 1, dtype=torch.int64, device=dev)
    sc = torch.empty(R * k + 1, dtype=torch.float32, device=dev)
    lib = skip.load_library()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    P = ctypes.c_void_p
    cp, rp, ip, sp = corpus.data_ptr(), regions.data_ptr(), ids.data_ptr(), sc.data_ptr()
    good = (cp, rp, ip, sp)
    for shift in ((2, 0, 0, 0), (8, 0, 0, 0), (0, 1, 0, 0), (0, 0, 4, 0), (0, 0, 0, 2)):
        c, r, i, s = (a + b for a, b in zip(good, shift))
        st = lib.skip_retrieve_regions_noalloc(P(c), N, d, skip.SKIP_BF16, None, P(r), R, k, P(i), P(s), stream)
        assert st == skip.SKIP_EINVAL, shift
    st = lib.skip_retrieve_regions_noalloc(P(cp), N, d, skip.SKIP_BF16, None, P(rp), R, k, P(ip), P(sp), stream)
    assert st == skip.SKIP_OK
    torch.cuda.synchronize()


def test_noalloc_binding_checks_tensors():
    dev = torch.device("cuda")
    corpus = synth.random_bf16(2000, 64, seed=5).to(dev)
    regions = synth.random_bf16(4, 64, seed=6).to(dev)
    ids = torch.empty(4, 7, dtype=torch.int64, device=dev)
    sc = torch.empty(4, 7, dtype=torch.float32, device=dev)
    bad_calls = [
        (corpus.float(), regions, ids, sc, None),                       # fp32 corpus
        (corpus, regions.float(), ids, sc, None),                       # fp32 regions
        (corpus, regions[:, :32], ids, sc, None),                       # d mismatch
        (corpus, regions.t().contiguous().t(), ids, sc, None),          # non-contiguous regions
        (corpus, regions, ids[:, :5], sc, None),                        # ids too small
        (corpus, regions, ids.int(), sc, None),                         # ids int32
        (corpus, regions, ids, sc.double(), None),                      # scores fp64
        (corpus.view(torch.uint8)[:, :64], regions, ids, sc, None),     # e4m3 without scales
        (corpus, regions, ids, sc, torch.ones(2000, device=dev)),       # bf16 with scales
    ]
    for c, r, i, s, scale in bad_calls:
        with pytest.raises((ValueError, TypeError)):
            skip.skip_retrieve_regions_noalloc(c, r, 7, i, s, row_scale=scale)
