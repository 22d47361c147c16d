"""CPU checks of the CUDA library: it builds for sm_103a, loads, exports every
entry point that include/*.h declares, and rejects bad arguments before any
device work.  No kernel runs here (there is no GPU in this container)."""
import ctypes
import glob
import os
import re

import pytest

import paper_2607_25422_gb300 as skip

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        names |= set(re.findall(r"SKIP_API\s+[\w\s\*]*?\b(skip_\w+)\s*\(", text))
    return sorted(names)


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("skip_corpus_load", "skip_corpus_free", "skip_retrieve", "skip_retrieve_regions",
              "skip_retrieve_host", "skip_sync_status", "skip_status_string"):
        assert n in names


def test_library_exports_every_declared_symbol():
    lib = skip.load_library()
    assert os.path.dirname(skip.library_path()).startswith(os.path.join(ROOT, "paper_2607_25422_gb300"))
    for n in declared_functions():
        assert hasattr(lib, n), n


def test_status_strings():
    for st in range(6):
        assert skip.skip_status_string(st)
    assert skip.skip_status_string(99) == "unknown status"


def test_load_rejects_bad_arguments_without_a_device():
    lib = skip.load_library()
    h = ctypes.c_void_p()
    buf = (ctypes.c_uint16 * 64)()
    # d not a multiple of 16, N < 1, e4m3 without scales, bf16 with scales.
    assert lib.skip_corpus_load(buf, 0, 2, 24, 0, None, None, ctypes.byref(h)) == skip.SKIP_EINVAL
    assert lib.skip_corpus_load(buf, 0, 0, 16, 0, None, None, ctypes.byref(h)) == skip.SKIP_EINVAL
    assert lib.skip_corpus_load(buf, 0, 2, 16, 1, None, None, ctypes.byref(h)) == skip.SKIP_EINVAL
    sc = (ctypes.c_float * 2)()
    assert lib.skip_corpus_load(buf, 0, 2, 16, 0, sc, None, ctypes.byref(h)) == skip.SKIP_EINVAL
    assert lib.skip_corpus_load(buf, 0, 1 << 31, 16, 0, None, None, ctypes.byref(h)) == skip.SKIP_EINVAL


@pytest.mark.skipif(os.path.exists("/dev/nvidia0"), reason="only meaningful without a GPU")
def test_load_without_gpu_is_unsupported_not_a_cpu_fallback():
    lib = skip.load_library()
    h = ctypes.c_void_p()
    buf = (ctypes.c_uint16 * 64)()
    assert lib.skip_corpus_load(buf, 0, 4, 16, 0, None, None, ctypes.byref(h)) == skip.SKIP_EUNSUPPORTED
    assert not h.value


def test_null_handles():
    lib = skip.load_library()
    assert lib.skip_corpus_free(None) == skip.SKIP_OK
    assert lib.skip_retrieve(None, None, None, 0, 0, 1, 1, None, None, None) == skip.SKIP_EINVAL
    assert lib.skip_sync_status(None, None) == skip.SKIP_EINVAL
    assert lib.skip_corpus_set_option(None, 0, 0) == skip.SKIP_EINVAL


def test_header_constants_match_the_binding():
    """Every `SKIP_NAME = value` of the C headers (status codes, options,
    paths) has the same value in the Python binding."""
    found = {}
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        for name, val in re.findall(r"\b(SKIP_[A-Z0-9_]+)\s*=\s*(\d+)", open(h).read()):
            found[name] = int(val)
    for name in ("SKIP_OK", "SKIP_EINVAL", "SKIP_ETIMEOUT", "SKIP_OPT_PATH", "SKIP_OPT_BOUND",
                 "SKIP_OPT_IVF_SPLIT", "SKIP_PATH_LATENCY"):
        assert name in found, name
    for name, val in found.items():
        assert getattr(skip, name) == val, name


def test_ivfpq_entry_points_reject_null_handles():
    lib = skip.load_library()
    assert lib.skip_ivfpq_set_option(None, skip.SKIP_OPT_IVF_SPLIT, 0) == skip.SKIP_EINVAL
    assert lib.skip_ivfpq_sync_status(None, None) == skip.SKIP_EINVAL
    assert lib.skip_ivfpq_info(None, None, None, None, None) == skip.SKIP_EINVAL
    assert lib.skip_ivfpq_lists(None, None, None, None, None) == skip.SKIP_EINVAL
    h = ctypes.c_void_p()
    # no centroids, codebook or offsets: refused before any device work
    assert lib.skip_ivfpq_load(None, 4, 64, None, 16, None, None, None, 0, None, ctypes.byref(h)) == skip.SKIP_EINVAL
    assert not h.value
