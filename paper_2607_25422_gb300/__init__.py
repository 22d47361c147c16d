"""Python binding of the GB300 region-conditional sparse retrieval library.

The functions carry the names of the C ABI in ``include/skip_retrieve.h`` and
only marshal arguments: tensors are handed over as raw pointers and streams
as ``cudaStream_t`` values; every step of the retrieval runs in the CUDA
library (``_build/libskip_retrieve.so``, built from ``csrc/`` for sm_103a).
There is no CPU path: if the library cannot be built or loaded, or the
device is not an sm_103 GPU, the calls raise.

The operation (paper §3.3 Eq. rcsr; App. B.2 Def. B.2; Alg. 1 RCSR loop and
Dedup): each region query is scored against the corpus by inner product, the
top-k_region ids are kept per region, and each question's region lists are
merged into a deduplicated top-K (max score per id, ties to the lower id).
The SKV passage gate (App. B.4 Def. B.4; ``include/skip_skv.h``) then keeps
the passages whose verification score nu reaches tau, at most
ceil(rho |K|) of them.  The IVF-PQ variant (``include/skip_ivfpq.h``) builds
and searches an inverted-file, product-quantised index of the corpus; QVS
(``include/skip_qvs.h``) scores and prunes visual tokens before retrieval;
BSCA (``include/skip_bsca.h``) fuses the kept tokens with the verified
chunks by attention over a sparse bipartite graph.
"""
from __future__ import annotations

import ctypes
import json
from typing import Optional

import torch

from . import _build

SKIP_BF16, SKIP_E4M3 = 0, 1
SKIP_OK, SKIP_EINVAL, SKIP_ENOMEM, SKIP_EUNSUPPORTED, SKIP_ETIMEOUT, SKIP_ECUDA, SKIP_ECANARY = range(7)
(SKIP_OPT_PATH, SKIP_OPT_WAIT_TIMEOUT_NS, SKIP_OPT_GRID, SKIP_OPT_TIMING, SKIP_OPT_CLUSTER, SKIP_OPT_MMA,
 SKIP_OPT_BOUND, SKIP_OPT_IVF_SPLIT, SKIP_OPT_CANARY, SKIP_OPT_RESIDENT, SKIP_OPT_IVF_REFINE) = range(11)
SKIP_PATH_AUTO, SKIP_PATH_TENSOR, SKIP_PATH_WARP, SKIP_PATH_LATENCY = range(4)
SKIP_MAX_K_REGION, SKIP_MAX_K = 1024, 2048

_lib = None


class SkvMlp(ctypes.Structure):
    """``skip_skv_mlp_t``: the gate MLP h_psi, pointers to device weights."""
    _fields_ = [("hidden", ctypes.c_int32), ("w1", ctypes.c_void_p), ("b1", ctypes.c_void_p),
                ("w2", ctypes.c_void_p), ("b2", ctypes.c_float)]


class SkipError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__("%s: %s (%d)" % (where, skip_status_string(status), status))


def library_path() -> str:
    return _build.LIB


def load_library():
    """Build (if stale) and load the CUDA library; raises if either fails."""
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(_build.build())
    P, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    lib.skip_corpus_load.argtypes = [P, ctypes.c_int, i64, i32, ctypes.c_int, P, P, ctypes.POINTER(P)]
    lib.skip_corpus_free.argtypes = [P]
    lib.skip_corpus_set_option.argtypes = [P, ctypes.c_int, i64]
    lib.skip_retrieve.argtypes = [P, P, P, i32, i32, i32, i32, P, P, P]
    lib.skip_retrieve_regions.argtypes = [P, P, i32, i32, P, P, P]
    lib.skip_retrieve_host.argtypes = [P, P, P, i32, i32, i32, i32, P, P, P]
    lib.skip_sync_status.argtypes = [P, P]
    lib.skip_last_plan.argtypes = [P, ctypes.c_char_p, i32]
    lib.skip_timing_report.argtypes = [P, ctypes.c_char_p, i32]
    lib.skip_retrieve_regions_noalloc.argtypes = [P, i64, i32, ctypes.c_int, P, P, i32, i32, P, P, P]
    lib.skip_skv_gate.argtypes = [P, P, i32, i32, P, P, ctypes.POINTER(SkvMlp), ctypes.c_float,
                                  ctypes.c_float, P, P, P, P, P]
    lib.skip_retrieve_skv.argtypes = [P, P, P, i32, i32, i32, i32, P, P, ctypes.POINTER(SkvMlp), ctypes.c_float,
                                      ctypes.c_float, P, P, P, P, P, P]
    lib.skip_ivfpq_build.argtypes = [P, P, i32, P, i32, P, ctypes.POINTER(P)]
    lib.skip_ivfpq_load.argtypes = [P, i32, i32, P, i32, P, P, P, i64, P, ctypes.POINTER(P)]
    lib.skip_ivfpq_lists.argtypes = [P, P, P, P, P]
    lib.skip_ivfpq_info.argtypes = [P, ctypes.POINTER(i64), ctypes.POINTER(i32), ctypes.POINTER(i32),
                                    ctypes.POINTER(i32)]
    lib.skip_ivfpq_free.argtypes = [P]
    lib.skip_ivfpq_search_regions.argtypes = [P, P, i32, i32, i32, P, P, P]
    lib.skip_ivfpq_search.argtypes = [P, P, P, i32, i32, i32, i32, i32, P, P, P]
    lib.skip_ivfpq_sync_status.argtypes = [P, P]
    lib.skip_ivfpq_set_option.argtypes = [P, ctypes.c_int, i64]
    lib.skip_ivfpq_timing_report.argtypes = [P, ctypes.c_char_p, i32]
    lib.skip_qvs_create.argtypes = [P, P, P, i32, i32, i32, i32, P, ctypes.POINTER(P)]
    lib.skip_qvs_free.argtypes = [P]
    lib.skip_qvs_count.argtypes = [i32, ctypes.c_float]
    lib.skip_qvs_count.restype = i32
    lib.skip_qvs_prune.argtypes = [P, P, i32, i32, P, ctypes.c_float, P, P, P, P, P]
    lib.skip_qvs_sync_status.argtypes = [P, P]
    lib.skip_bsca_create.argtypes = [i32, i32, i32, i32, i32, ctypes.POINTER(P)]
    lib.skip_bsca_free.argtypes = [P]
    lib.skip_bsca_run.argtypes = [P, i32, P, P, i32, P, P, P, P, P, ctypes.c_float, P, P, P, P, P]
    lib.skip_bsca_sync_status.argtypes = [P, P]
    lib.skip_status_string.argtypes = [ctypes.c_int]
    lib.skip_status_string.restype = ctypes.c_char_p
    for f in ("skip_corpus_load", "skip_corpus_free", "skip_corpus_set_option", "skip_retrieve",
              "skip_retrieve_regions", "skip_retrieve_host", "skip_sync_status", "skip_last_plan",
              "skip_timing_report", "skip_retrieve_regions_noalloc", "skip_skv_gate", "skip_retrieve_skv",
              "skip_ivfpq_build", "skip_ivfpq_load", "skip_ivfpq_lists", "skip_ivfpq_info", "skip_ivfpq_free",
              "skip_ivfpq_search_regions", "skip_ivfpq_search", "skip_ivfpq_sync_status", "skip_ivfpq_set_option",
              "skip_ivfpq_timing_report", "skip_qvs_create", "skip_qvs_free", "skip_qvs_prune", "skip_qvs_sync_status",
              "skip_bsca_create", "skip_bsca_free", "skip_bsca_run", "skip_bsca_sync_status"):
        getattr(lib, f).restype = ctypes.c_int
    _lib = lib
    return lib


def skip_status_string(status: int) -> str:
    return load_library().skip_status_string(int(status)).decode()


def _check(status: int, where: str):
    if status != SKIP_OK:
        raise SkipError(status, where)


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


class Corpus:
    """A corpus handle (``skip_corpus_t``); the library owns the device copy."""

    def __init__(self, handle, N: int, d: int, dtype: int, device: torch.device):
        self.handle = handle
        self.N, self.d, self.dtype, self.device = N, d, dtype, device

    def free(self):
        if self.handle:
            load_library().skip_corpus_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass

    def set_option(self, option: int, value: int):
        skip_corpus_set_option(self, option, value)


def skip_corpus_load(rows: torch.Tensor, row_scale: Optional[torch.Tensor] = None,
                     stream=None) -> Corpus:
    """Copy a corpus into the library.  rows: [N, d] bfloat16 (or uint16 bf16
    bits), or uint8 / float8_e4m3fn bytes with row_scale [N] float32; on the
    host or on the current CUDA device."""
    lib = load_library()
    if rows.dim() != 2:
        raise ValueError("rows must be [N, d]")
    if rows.dtype in (torch.bfloat16, torch.uint16, torch.int16):
        dtype = SKIP_BF16
    elif rows.dtype in (torch.uint8, torch.float8_e4m3fn):
        dtype = SKIP_E4M3
    else:
        raise TypeError("rows must be bf16 or e4m3 bytes")
    rows = rows.contiguous()
    on_dev = rows.is_cuda
    if row_scale is not None:
        row_scale = row_scale.to(device=rows.device, dtype=torch.float32).contiguous()
    dev = rows.device if on_dev else torch.device("cuda", torch.cuda.current_device())
    h = ctypes.c_void_p()
    st = lib.skip_corpus_load(_ptr(rows), int(on_dev), rows.shape[0], rows.shape[1], dtype,
                              _ptr(row_scale), ctypes.c_void_p(_stream(stream)), ctypes.byref(h))
    _check(st, "skip_corpus_load")
    return Corpus(h, rows.shape[0], rows.shape[1], dtype, dev)


def skip_corpus_free(corpus: Corpus):
    corpus.free()


def skip_corpus_set_option(corpus: Corpus, option: int, value: int):
    _check(load_library().skip_corpus_set_option(corpus.handle, int(option), int(value)),
           "skip_corpus_set_option")


def _regions_arg(regions: torch.Tensor, corpus: Corpus) -> torch.Tensor:
    if regions.dim() != 2 or regions.shape[1] != corpus.d:
        raise ValueError("regions must be [R_total, d]")
    if regions.dtype not in (torch.bfloat16, torch.uint16, torch.int16):
        raise TypeError("regions must be bf16")
    return regions.contiguous()


def skip_retrieve(corpus: Corpus, regions: torch.Tensor, region_offsets: torch.Tensor,
                  k_region: int, K: int, out_ids: Optional[torch.Tensor] = None,
                  out_scores: Optional[torch.Tensor] = None, stream=None):
    """Whole path on device tensors; returns (ids int64 [Q, K], scores fp32 [Q, K])."""
    lib = load_library()
    regions = _regions_arg(regions, corpus)
    offs = region_offsets.to(device=regions.device, dtype=torch.int32).contiguous()
    Q = offs.numel() - 1
    if out_ids is None:
        out_ids = torch.empty(Q, K, dtype=torch.int64, device=regions.device)
    if out_scores is None:
        out_scores = torch.empty(Q, K, dtype=torch.float32, device=regions.device)
    st = lib.skip_retrieve(corpus.handle, _ptr(regions), _ptr(offs), Q, regions.shape[0], int(k_region),
                           int(K), _ptr(out_ids), _ptr(out_scores), ctypes.c_void_p(_stream(stream)))
    _check(st, "skip_retrieve")
    return out_ids, out_scores


def skip_retrieve_regions(corpus: Corpus, regions: torch.Tensor, k_region: int,
                          reg_ids: Optional[torch.Tensor] = None,
                          reg_scores: Optional[torch.Tensor] = None, stream=None):
    """Per-region step only; returns (ids int64 [R, k], scores fp32 [R, k])."""
    lib = load_library()
    regions = _regions_arg(regions, corpus)
    R = regions.shape[0]
    if reg_ids is None:
        reg_ids = torch.empty(R, k_region, dtype=torch.int64, device=regions.device)
    if reg_scores is None:
        reg_scores = torch.empty(R, k_region, dtype=torch.float32, device=regions.device)
    st = lib.skip_retrieve_regions(corpus.handle, _ptr(regions), R, int(k_region), _ptr(reg_ids),
                                   _ptr(reg_scores), ctypes.c_void_p(_stream(stream)))
    _check(st, "skip_retrieve_regions")
    return reg_ids, reg_scores


def skip_retrieve_host(corpus: Corpus, regions: torch.Tensor, region_offsets: torch.Tensor,
                       k_region: int, K: int, out_ids: Optional[torch.Tensor] = None,
                       out_scores: Optional[torch.Tensor] = None, stream=None):
    """Whole path on HOST tensors (pinned memory is fastest); blocks until done."""
    lib = load_library()
    if regions.is_cuda:
        raise ValueError("skip_retrieve_host takes host tensors")
    regions = _regions_arg(regions, corpus)
    offs = region_offsets.to(dtype=torch.int32).contiguous()
    Q = offs.numel() - 1
    if out_ids is None:
        out_ids = torch.empty(Q, K, dtype=torch.int64)
    if out_scores is None:
        out_scores = torch.empty(Q, K, dtype=torch.float32)
    st = lib.skip_retrieve_host(corpus.handle, _ptr(regions), _ptr(offs), Q, regions.shape[0],
                                int(k_region), int(K), _ptr(out_ids), _ptr(out_scores),
                                ctypes.c_void_p(_stream(stream)))
    _check(st, "skip_retrieve_host")
    return out_ids, out_scores


def skip_retrieve_regions_noalloc(corpus_rows: torch.Tensor, regions: torch.Tensor, k_region: int,
                                  reg_ids: torch.Tensor, reg_scores: torch.Tensor,
                                  row_scale: Optional[torch.Tensor] = None, stream=None):
    """Per-region step on caller-owned device tensors, with no device
    allocation by the library (its scratch is a fixed array in the library's
    device memory).  For callers whose device memory must all come from
    their own pool; the output tensors are theirs to allocate."""
    lib = load_library()
    if not (corpus_rows.is_cuda and regions.is_cuda and reg_ids.is_cuda and reg_scores.is_cuda):
        raise ValueError("skip_retrieve_regions_noalloc takes device tensors")
    if corpus_rows.dim() != 2:
        raise ValueError("corpus_rows must be [N, d]")
    if corpus_rows.dtype in (torch.bfloat16, torch.uint16, torch.int16):
        dtype = SKIP_BF16
        if row_scale is not None:
            raise ValueError("a bf16 corpus takes no row_scale")
    elif corpus_rows.dtype in (torch.uint8, torch.float8_e4m3fn):
        dtype = SKIP_E4M3
        if row_scale is None or row_scale.dtype != torch.float32 or not row_scale.is_cuda \
                or row_scale.shape != (corpus_rows.shape[0],) or not row_scale.is_contiguous():
            raise ValueError("an e4m3 corpus needs row_scale: contiguous float32 [N] on the device")
    else:
        raise TypeError("corpus_rows must be bf16 (or uint16 bits) or e4m3 bytes (uint8 / float8_e4m3fn)")
    if not corpus_rows.is_contiguous():
        raise ValueError("corpus_rows must be contiguous")
    if regions.dim() != 2 or regions.shape[1] != corpus_rows.shape[1]:
        raise ValueError("regions must be [R_total, d] with the corpus's d")
    if regions.dtype not in (torch.bfloat16, torch.uint16, torch.int16) or not regions.is_contiguous():
        raise TypeError("regions must be contiguous bf16")
    R = regions.shape[0]
    if reg_ids.dtype != torch.int64 or tuple(reg_ids.shape) != (R, int(k_region)) or not reg_ids.is_contiguous():
        raise ValueError("reg_ids must be contiguous int64 [R_total, k_region]")
    if reg_scores.dtype != torch.float32 or tuple(reg_scores.shape) != (R, int(k_region)) \
            or not reg_scores.is_contiguous():
        raise ValueError("reg_scores must be contiguous float32 [R_total, k_region]")
    st = lib.skip_retrieve_regions_noalloc(_ptr(corpus_rows), corpus_rows.shape[0], corpus_rows.shape[1], dtype,
                                           _ptr(row_scale), _ptr(regions), regions.shape[0], int(k_region),
                                           _ptr(reg_ids), _ptr(reg_scores), ctypes.c_void_p(_stream(stream)))
    _check(st, "skip_retrieve_regions_noalloc")
    return reg_ids, reg_scores


def _skv_mlp(w1: torch.Tensor, b1: torch.Tensor, w2: torch.Tensor, b2: float):
    """Marshal the gate weights (device tensors, kept alive by the caller)."""
    if w1.dtype not in (torch.bfloat16, torch.uint16, torch.int16) or b1.dtype != torch.float32 \
            or w2.dtype != torch.float32:
        raise TypeError("w1 must be bf16 [H, 5d]; b1, w2 float32 [H]")
    if not (w1.is_contiguous() and b1.is_contiguous() and w2.is_contiguous()):
        raise ValueError("gate weights must be contiguous")
    return SkvMlp(w1.shape[0], w1.data_ptr(), b1.data_ptr(), w2.data_ptr(), float(b2))


def skip_skv_gate(corpus: Corpus, cand_ids: torch.Tensor, qbar: torch.Tensor, vbar: torch.Tensor,
                  w1: torch.Tensor, b1: torch.Tensor, w2: torch.Tensor, b2: float, tau_nu: float = 0.5,
                  rho_r: float = 0.6, with_nu_all: bool = False, stream=None):
    """SKV gate on candidate lists (device int64 [Q, K], -1 = empty).
    Returns (ids int64 [Q, K], nu fp32 [Q, K], count int32 [Q]) and, with
    with_nu_all, nu of every input slot as a fourth tensor."""
    lib = load_library()
    cand_ids = cand_ids.to(torch.int64).contiguous()
    Q, K = cand_ids.shape
    dev = cand_ids.device
    qbar, vbar = qbar.contiguous(), vbar.contiguous()
    mlp = _skv_mlp(w1, b1, w2, b2)
    out_ids = torch.empty(Q, K, dtype=torch.int64, device=dev)
    out_nu = torch.empty(Q, K, dtype=torch.float32, device=dev)
    count = torch.empty(Q, dtype=torch.int32, device=dev)
    nu_all = torch.empty(Q, K, dtype=torch.float32, device=dev) if with_nu_all else None
    st = lib.skip_skv_gate(corpus.handle, _ptr(cand_ids), Q, K, _ptr(qbar), _ptr(vbar), ctypes.byref(mlp),
                           float(tau_nu), float(rho_r), _ptr(out_ids), _ptr(out_nu), _ptr(count), _ptr(nu_all),
                           ctypes.c_void_p(_stream(stream)))
    _check(st, "skip_skv_gate")
    return (out_ids, out_nu, count, nu_all) if with_nu_all else (out_ids, out_nu, count)


def skip_retrieve_skv(corpus: Corpus, regions: torch.Tensor, region_offsets: torch.Tensor, k_region: int,
                      K: int, qbar: torch.Tensor, vbar: torch.Tensor, w1: torch.Tensor, b1: torch.Tensor,
                      w2: torch.Tensor, b2: float, tau_nu: float = 0.5, rho_r: float = 0.6,
                      with_merged: bool = False, stream=None):
    """Retrieval and gate in one call.  Returns (ids, nu, count) and, with
    with_merged, the merged lists (ids int64 [Q, K], scores fp32 [Q, K])."""
    lib = load_library()
    regions = _regions_arg(regions, corpus)
    offs = region_offsets.to(device=regions.device, dtype=torch.int32).contiguous()
    Q = offs.numel() - 1
    dev = regions.device
    mlp = _skv_mlp(w1, b1, w2, b2)
    out_ids = torch.empty(Q, K, dtype=torch.int64, device=dev)
    out_nu = torch.empty(Q, K, dtype=torch.float32, device=dev)
    count = torch.empty(Q, dtype=torch.int32, device=dev)
    m_ids = torch.empty(Q, K, dtype=torch.int64, device=dev) if with_merged else None
    m_sc = torch.empty(Q, K, dtype=torch.float32, device=dev) if with_merged else None
    st = lib.skip_retrieve_skv(corpus.handle, _ptr(regions), _ptr(offs), Q, regions.shape[0], int(k_region),
                               int(K), _ptr(qbar.contiguous()), _ptr(vbar.contiguous()), ctypes.byref(mlp),
                               float(tau_nu), float(rho_r), _ptr(out_ids), _ptr(out_nu), _ptr(count),
                               _ptr(m_ids), _ptr(m_sc), ctypes.c_void_p(_stream(stream)))
    _check(st, "skip_retrieve_skv")
    return (out_ids, out_nu, count, m_ids, m_sc) if with_merged else (out_ids, out_nu, count)


class IvfIndex:
    """An IVF-PQ index handle (``skip_ivfpq_t``)."""

    def __init__(self, handle):
        self.handle = handle
        lib = load_library()
        N, d, C, M = ctypes.c_int64(), ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
        _check(lib.skip_ivfpq_info(handle, ctypes.byref(N), ctypes.byref(d), ctypes.byref(C), ctypes.byref(M)),
               "skip_ivfpq_info")
        self.N, self.d, self.C, self.M = N.value, d.value, C.value, M.value

    def free(self):
        if self.handle:
            load_library().skip_ivfpq_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass

    def set_option(self, option: int, value: int):
        _check(load_library().skip_ivfpq_set_option(self.handle, int(option), int(value)), "skip_ivfpq_set_option")


def skip_ivfpq_build(corpus: Corpus, centroids: torch.Tensor, codebook: torch.Tensor, stream=None) -> IvfIndex:
    """Index of a loaded bf16 corpus: centroids bf16 [C, d], codebook float32
    [M, 256, d / M] (device tensors)."""
    lib = load_library()
    centroids, codebook = centroids.contiguous(), codebook.to(torch.float32).contiguous()
    h = ctypes.c_void_p()
    st = lib.skip_ivfpq_build(corpus.handle, _ptr(centroids), centroids.shape[0], _ptr(codebook), codebook.shape[0],
                              ctypes.c_void_p(_stream(stream)), ctypes.byref(h))
    _check(st, "skip_ivfpq_build")
    return IvfIndex(h)


def skip_ivfpq_load(centroids: torch.Tensor, codebook: torch.Tensor, list_offsets: torch.Tensor, ids: torch.Tensor,
                    codes: torch.Tensor, stream=None) -> IvfIndex:
    """Index from device arrays: offsets int64 [C + 1], ids int32 [N] and codes
    uint8 [N, M] in list order."""
    lib = load_library()
    centroids, codebook = centroids.contiguous(), codebook.to(torch.float32).contiguous()
    list_offsets = list_offsets.to(torch.int64).contiguous()
    ids, codes = ids.to(torch.int32).contiguous(), codes.to(torch.uint8).contiguous()
    h = ctypes.c_void_p()
    st = lib.skip_ivfpq_load(_ptr(centroids), centroids.shape[0], centroids.shape[1], _ptr(codebook), codebook.shape[0],
                             _ptr(list_offsets), _ptr(ids), _ptr(codes), ids.shape[0],
                             ctypes.c_void_p(_stream(stream)), ctypes.byref(h))
    _check(st, "skip_ivfpq_load")
    return IvfIndex(h)


def skip_ivfpq_lists(index: IvfIndex, device=None, stream=None):
    """(offsets int64 [C + 1], ids int32 [N], codes uint8 [N, M]) on the device."""
    device = device or torch.device("cuda", torch.cuda.current_device())
    off = torch.empty(index.C + 1, dtype=torch.int64, device=device)
    ids = torch.empty(index.N, dtype=torch.int32, device=device)
    codes = torch.empty(index.N, index.M, dtype=torch.uint8, device=device)
    _check(load_library().skip_ivfpq_lists(index.handle, _ptr(off), _ptr(ids), _ptr(codes),
                                          ctypes.c_void_p(_stream(stream))), "skip_ivfpq_lists")
    return off, ids, codes


def skip_ivfpq_search_regions(index: IvfIndex, regions: torch.Tensor, nprobe: int, k_region: int, stream=None):
    """Per region: (ids int64 [R, k], scores fp32 [R, k])."""
    regions = regions.contiguous()
    R = regions.shape[0]
    ids = torch.empty(R, k_region, dtype=torch.int64, device=regions.device)
    sc = torch.empty(R, k_region, dtype=torch.float32, device=regions.device)
    _check(load_library().skip_ivfpq_search_regions(index.handle, _ptr(regions), R, int(nprobe), int(k_region),
                                                    _ptr(ids), _ptr(sc), ctypes.c_void_p(_stream(stream))),
           "skip_ivfpq_search_regions")
    return ids, sc


def skip_ivfpq_search(index: IvfIndex, regions: torch.Tensor, region_offsets: torch.Tensor, nprobe: int,
                      k_region: int, K: int, out_ids: Optional[torch.Tensor] = None,
                      out_scores: Optional[torch.Tensor] = None, stream=None):
    """Per region, then per question: (ids int64 [Q, K], scores fp32 [Q, K])."""
    regions = regions.contiguous()
    offs = region_offsets.to(device=regions.device, dtype=torch.int32).contiguous()
    Q = offs.numel() - 1
    if out_ids is None:
        out_ids = torch.empty(Q, K, dtype=torch.int64, device=regions.device)
    if out_scores is None:
        out_scores = torch.empty(Q, K, dtype=torch.float32, device=regions.device)
    _check(load_library().skip_ivfpq_search(index.handle, _ptr(regions), _ptr(offs), Q, regions.shape[0], int(nprobe),
                                            int(k_region), int(K), _ptr(out_ids), _ptr(out_scores),
                                            ctypes.c_void_p(_stream(stream))), "skip_ivfpq_search")
    return out_ids, out_scores


def skip_ivfpq_sync_status(index: IvfIndex, stream=None) -> int:
    return int(load_library().skip_ivfpq_sync_status(index.handle, ctypes.c_void_p(_stream(stream))))


def skip_ivfpq_timing_report(index: IvfIndex) -> dict:
    buf = ctypes.create_string_buffer(1 << 16)
    _check(load_library().skip_ivfpq_timing_report(index.handle, buf, 1 << 16), "skip_ivfpq_timing_report")
    return json.loads(buf.value.decode())


class QvsHead:
    """A QVS head (``skip_qvs_t``): weights copied to the library."""

    def __init__(self, handle, d, dk):
        self.handle, self.d, self.dk = handle, d, dk

    def free(self):
        if self.handle:
            load_library().skip_qvs_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def skip_qvs_create(wv: torch.Tensor, bv: Optional[torch.Tensor], wb: torch.Tensor, max_images: int,
                    max_tokens: int, stream=None) -> QvsHead:
    """QVS head from device tensors: wv bf16 [d_k, d], bv float32 [d_k] or None, wb float32 [d]."""
    wv = wv.contiguous()
    bv = None if bv is None else bv.to(torch.float32).contiguous()
    wb = wb.to(torch.float32).contiguous()
    h = ctypes.c_void_p()
    st = load_library().skip_qvs_create(_ptr(wv), _ptr(bv), _ptr(wb), wv.shape[1], wv.shape[0], int(max_images),
                                        int(max_tokens), ctypes.c_void_p(_stream(stream)), ctypes.byref(h))
    _check(st, "skip_qvs_create")
    return QvsHead(h, wv.shape[1], wv.shape[0])


def skip_qvs_count(L: int, rho_v: float) -> int:
    return int(load_library().skip_qvs_count(int(L), float(rho_v)))


def skip_qvs_prune(head: QvsHead, tokens: torch.Tensor, fq: torch.Tensor, rho_v: float, with_tokens: bool = False,
                   with_logits: bool = False, stream=None):
    """tokens bf16 [B, L, d], fq bf16 [B, d_k] (device).  Returns (idx int32
    [B, n], score fp32 [B, n]) plus the kept tokens [B, n, d] and / or all
    logits [B, L] when asked."""
    tokens, fq = tokens.contiguous(), fq.contiguous()
    B, L, d = tokens.shape
    n = skip_qvs_count(L, rho_v)
    dev = tokens.device
    idx = torch.empty(B, n, dtype=torch.int32, device=dev)
    score = torch.empty(B, n, dtype=torch.float32, device=dev)
    kept = torch.empty(B, n, d, dtype=tokens.dtype, device=dev) if with_tokens else None
    logits = torch.empty(B, L, dtype=torch.float32, device=dev) if with_logits else None
    st = load_library().skip_qvs_prune(head.handle, _ptr(tokens), B, L, _ptr(fq), float(rho_v), _ptr(idx),
                                       _ptr(score), _ptr(kept), _ptr(logits), ctypes.c_void_p(_stream(stream)))
    _check(st, "skip_qvs_prune")
    out = [idx, score]
    if with_tokens:
        out.append(kept)
    if with_logits:
        out.append(logits)
    return tuple(out)


class BscaHandle:
    """A BSCA workspace (``skip_bsca_t``)."""

    def __init__(self, handle, dp, dh, dout):
        self.handle, self.dp, self.dh, self.dout = handle, dp, dh, dout

    def free(self):
        if self.handle:
            load_library().skip_bsca_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def skip_bsca_create(d_p: int, d_h: int, d_o: int, max_questions: int, max_tokens: int) -> BscaHandle:
    h = ctypes.c_void_p()
    _check(load_library().skip_bsca_create(int(d_p), int(d_h), int(d_o), int(max_questions), int(max_tokens),
                                           ctypes.byref(h)), "skip_bsca_create")
    return BscaHandle(h, d_p, d_h, d_o)


def skip_bsca_run(handle: BscaHandle, vis_offsets: torch.Tensor, chunk_offsets: torch.Tensor, hv: torch.Tensor,
                  qh: torch.Tensor, hk: torch.Tensor, kh: torch.Tensor, vh: torch.Tensor, dbar: float = 4.0,
                  with_graph: bool = False, stream=None):
    """Device tensors (bf16 projections, int32 offsets).  Returns out fp32
    [Nv, d_o] and, with with_graph, (degree int32 [Nv], edges int64 [Nv]
    neighbour bit masks, tau_e fp32 [Q])."""
    vo = vis_offsets.to(torch.int32).contiguous()
    co = chunk_offsets.to(torch.int32).contiguous()
    hv, qh, hk, kh, vh = (t.contiguous() for t in (hv, qh, hk, kh, vh))
    Q = vo.numel() - 1
    Nv = hv.shape[0]
    out = torch.empty(Nv, handle.dout, dtype=torch.float32, device=hv.device)
    deg = torch.empty(Nv, dtype=torch.int32, device=hv.device) if with_graph else None
    tau = torch.empty(Q, dtype=torch.float32, device=hv.device) if with_graph else None
    edges = torch.empty(Nv, dtype=torch.int64, device=hv.device) if with_graph else None
    _check(load_library().skip_bsca_run(handle.handle, Q, _ptr(vo), _ptr(co), Nv, _ptr(hv), _ptr(qh), _ptr(hk),
                                        _ptr(kh), _ptr(vh), float(dbar), _ptr(out), _ptr(deg), _ptr(edges), _ptr(tau),
                                        ctypes.c_void_p(_stream(stream))), "skip_bsca_run")
    return (out, deg, edges, tau) if with_graph else out


def skip_qvs_sync_status(head: QvsHead, stream=None) -> int:
    return int(load_library().skip_qvs_sync_status(head.handle, ctypes.c_void_p(_stream(stream))))


def skip_bsca_sync_status(handle: BscaHandle, stream=None) -> int:
    return int(load_library().skip_bsca_sync_status(handle.handle, ctypes.c_void_p(_stream(stream))))


def skip_sync_status(corpus: Corpus, stream=None) -> int:
    """Synchronise and return the status latched by the kernels (SKIP_OK, ...)."""
    return int(load_library().skip_sync_status(corpus.handle, ctypes.c_void_p(_stream(stream))))


def skip_last_plan(corpus: Corpus) -> dict:
    buf = ctypes.create_string_buffer(1024)
    _check(load_library().skip_last_plan(corpus.handle, buf, 1024), "skip_last_plan")
    return json.loads(buf.value.decode())


def skip_timing_report(corpus: Corpus) -> dict:
    """Per-kernel launches and device ms accumulated since the last report
    (needs SKIP_OPT_TIMING = 1); clears the record."""
    buf = ctypes.create_string_buffer(1 << 16)
    _check(load_library().skip_timing_report(corpus.handle, buf, 1 << 16), "skip_timing_report")
    return json.loads(buf.value.decode())


__all__ = [n for n in dir() if n.startswith("skip_") or n.startswith("SKIP_")] + [
    "Corpus", "SkipError", "SkvMlp", "IvfIndex", "QvsHead", "BscaHandle", "load_library", "library_path"]
