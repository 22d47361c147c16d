"""The allocation-free per-region entry point against the handle-based one.

skip_retrieve_regions_noalloc serves callers that cannot let a library
allocate device memory -- applications whose framework owns every device
allocation, and serving loops that cannot take cudaMalloc's device-wide
synchronisation.  Its scratch is a fixed array in the library's device
memory, shared by all calls on a device.  This test calls it twice in a row
through the C ABI (the second call finds the previous call's leftovers in
that array) and compares both results with skip_retrieve_regions on the
same inputs, within the parity tolerance of the other tests.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2607_25422_gb300 as skip
import synth

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
        _same(ids.cpu().numpy(), sc.cpu().numpy(), ref_ids, ref_sc)


def test_noalloc_rejects_sizes_beyond_its_scratch():
    dev = torch.device("cuda")
    corpus = synth.random_bf16(5000, 64, seed=1).to(dev)
    regions = synth.random_bf16(4000, 64, seed=2).to(dev)
    ids = torch.empty(4000, 1000, dtype=torch.int64, device=dev)
    sc = torch.empty(4000, 1000, dtype=torch.float32, device=dev)
    with pytest.raises(skip.SkipError) as e:
        skip.skip_retrieve_regions_noalloc(corpus, regions, 1000, ids, sc)
    assert e.value.status == skip.SKIP_EUNSUPPORTED
