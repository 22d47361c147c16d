"""CPU oracle for region-conditional sparse retrieval (test infrastructure).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg call this module; the product path never does.
It shares no code with the CUDA library.  The arithmetic lives in
``rcsr_oracle.c`` (fp64, plain loops, one OpenMP thread per region); this
file only compiles it with gcc and marshals numpy arrays.

Functions and what they follow:

* ``region_topk``  -- Def. B.2 MIPS(q_{r_i}, D; k_r) / Eq. rcsr top-k':
  exact per-region top-k by (score desc, id asc).
* ``merge``        -- §3.3 / Def. B.2 / Alg. 1 Dedup of the union of the
  per-region lists, keeping each id's max score, cut to the first K.
* ``retrieve``     -- both steps (the CPU baseline).
* ``score_matrix`` -- every s(r, i) in fp64 (brute force on tiny inputs).
* ``scores_at``    -- s(r, i) at chosen (region, id) pairs.
* ``skv``          -- App. B.4 Def. B.4 (Eq. skv_score) and the Alg. 1 TopK
  after it: the passage gate nu_j = sigmoid(h_psi(features)), kept when
  nu_j >= tau, the best ceil(rho |K|) by (nu desc, id asc)
  (``skv_oracle.c``).
* ``bf16_round``   -- a double rounded to bf16 (ties to even), as bits.
* ``ivf_assign``, ``pq_encode``, ``ivfpq_build``, ``ivfpq_search``,
  ``ivfpq_search_refine``, ``ivfpq_scores_at`` -- the IVF-PQ index (§4.1 "Implementation", App. I.4;
  the published inverted file with product-quantised residuals and
  asymmetric inner-product scoring) and its search (``ivfpq_oracle.c``).
* ``qvs``, ``qvs_count`` -- App. B.1 Def. B.1 (Eq. qvs_score) and the Alg. 1
  QVS prune: token scores sigmoid(<f_q, W_v v + b_v> / sqrt(d_k) + <w_b, v>)
  and the top ceil(rho_v L) tokens (``qvs_oracle.c``).
* ``bsca``, ``bsca_edges_count`` -- App. B.3 Def. B.3 (Eq. bsca_edges,
  bsca_attn): the bipartite edge set by cosine threshold and the attention of
  each visual token over its chunk neighbours (``bsca_oracle.c``).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRCS = [os.path.join(_HERE, "rcsr_oracle.c"), os.path.join(_HERE, "skv_oracle.c"),
         os.path.join(_HERE, "ivfpq_oracle.c"), os.path.join(_HERE, "qvs_oracle.c"),
         os.path.join(_HERE, "bsca_oracle.c")]
_OUT = os.path.join(_HERE, "_build", "libskip_oracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP) into oracle/_build/."""
    if not force and os.path.exists(_OUT) and all(os.path.getmtime(_OUT) >= os.path.getmtime(f)
                                                   for f in _SRCS):
        return _OUT
    os.makedirs(os.path.dirname(_OUT), exist_ok=True)
    tmp = _OUT + ".tmp.%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-Wall", "-Wextra",
           *_SRCS, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _OUT)
    return _OUT


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(build())
    P = ctypes.c_void_p
    i64, i32 = ctypes.c_int64, ctypes.c_int
    lib.skip_oracle_region_topk.argtypes = [P, P, P, i64, i32, P, i64, i32, P, P, i32]
    lib.skip_oracle_merge.argtypes = [P, P, i32, i32, P, i32, i32, P, P]
    lib.skip_oracle_retrieve.argtypes = [P, P, P, i64, i32, P, P, i32, i64, i32, i32, P, P, P, P, i32]
    lib.skip_oracle_score_matrix.argtypes = [P, P, P, i64, i32, P, i64, P]
    lib.skip_oracle_scores_at.argtypes = [P, P, P, i64, i32, P, P, P, i64, P]
    lib.skip_oracle_bf16_value.argtypes = [ctypes.c_uint16]
    lib.skip_oracle_bf16_value.restype = ctypes.c_double
    lib.skip_oracle_e4m3_value.argtypes = [ctypes.c_uint8]
    lib.skip_oracle_e4m3_value.restype = ctypes.c_double
    lib.skip_oracle_skv.argtypes = [P, i64, i32, P, i32, i32, P, P, P, P, P, ctypes.c_float, i32,
                                    ctypes.c_double, ctypes.c_double, P, P, P, P, P]
    lib.skip_oracle_skv_count.argtypes = [i32, ctypes.c_double]
    lib.skip_oracle_bf16_round.argtypes = [ctypes.c_double]
    lib.skip_oracle_bf16_round.restype = ctypes.c_uint16
    lib.skip_oracle_ivf_assign.argtypes = [P, i64, i32, P, i32, P]
    lib.skip_oracle_pq_encode.argtypes = [P, i64, i32, P, P, P, i32, i32, P]
    lib.skip_oracle_ivfpq_search.argtypes = [P, i32, i32, P, P, P, P, i32, i32, P, i32, i32, i32, P, P, P]
    lib.skip_oracle_ivfpq_scores_at.argtypes = [P, i32, P, P, i64, P, i32, i32, P, P, P, i64, P]
    lib.skip_oracle_qvs.argtypes = [P, i32, i32, i32, P, P, P, P, i32, ctypes.c_double, P, P, P]
    lib.skip_oracle_bsca.argtypes = [P, P, i32, P, P, P, P, P, i32, i32, i32, i32, ctypes.c_double, P, P, P, P, P]
    lib.skip_oracle_bsca_edges_count.argtypes = [i32, ctypes.c_double]
    lib.skip_oracle_bsca.restype = ctypes.c_int
    lib.skip_oracle_bsca_edges_count.restype = ctypes.c_int
    lib.skip_oracle_qvs_count.argtypes = [i32, ctypes.c_double]
    for f in ("skip_oracle_qvs", "skip_oracle_qvs_count", "skip_oracle_ivf_assign", "skip_oracle_pq_encode",
              "skip_oracle_ivfpq_search",
              "skip_oracle_ivfpq_scores_at"):
        getattr(lib, f).restype = ctypes.c_int
    for f in ("skip_oracle_region_topk", "skip_oracle_merge", "skip_oracle_retrieve", "skip_oracle_skv",
              "skip_oracle_skv_count",
              "skip_oracle_score_matrix", "skip_oracle_scores_at", "skip_oracle_threads"):
        getattr(lib, f).restype = ctypes.c_int
    _lib = lib
    return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _corpus_args(corpus, row_scale):
    """corpus: uint16 [N, d] (bf16 bits) or uint8 [N, d] (e4m3 bytes)."""
    corpus = np.ascontiguousarray(corpus)
    if corpus.dtype == np.uint16:
        return corpus, None, None
    if corpus.dtype == np.uint8:
        if row_scale is None:
            raise ValueError("e4m3 corpus needs row_scale")
        return None, corpus, np.ascontiguousarray(row_scale, dtype=np.float32)
    raise TypeError("corpus must be uint16 (bf16 bits) or uint8 (e4m3)")


def threads() -> int:
    return int(_load().skip_oracle_threads())


def bf16_value(bits: int) -> float:
    return float(_load().skip_oracle_bf16_value(int(bits)))


def e4m3_value(byte: int) -> float:
    return float(_load().skip_oracle_e4m3_value(int(byte)))


def region_topk(corpus, regions, kk, row_scale=None, nthreads=0):
    """Exact top-kk per region: (ids int64 [R, kk], scores float64 [R, kk])."""
    lib = _load()
    cb, ce, sc = _corpus_args(corpus, row_scale)
    c = cb if cb is not None else ce
    regions = np.ascontiguousarray(regions, dtype=np.uint16)
    N, d = c.shape
    R = regions.shape[0]
    ids = np.empty((R, kk), dtype=np.int64)
    sco = np.empty((R, kk), dtype=np.float64)
    rc = lib.skip_oracle_region_topk(_ptr(cb), _ptr(ce), _ptr(sc), N, d, _ptr(regions), R, kk,
                                     _ptr(ids), _ptr(sco), int(nthreads))
    if rc:
        raise RuntimeError("oracle region_topk failed (%d)" % rc)
    return ids, sco


def merge(reg_ids, reg_scores, k, offsets, K):
    """Union + dedup (max score) + top-K per question: (ids [Q, K], scores [Q, K])."""
    lib = _load()
    reg_ids = np.ascontiguousarray(reg_ids, dtype=np.int64)
    reg_scores = np.ascontiguousarray(reg_scores, dtype=np.float64)
    offsets = np.ascontiguousarray(offsets, dtype=np.int32)
    Q = offsets.shape[0] - 1
    ld = reg_ids.shape[1] if reg_ids.ndim == 2 else k
    out_ids = np.empty((Q, K), dtype=np.int64)
    out_sc = np.empty((Q, K), dtype=np.float64)
    rc = lib.skip_oracle_merge(_ptr(reg_ids), _ptr(reg_scores), ld, k, _ptr(offsets), Q, K,
                               _ptr(out_ids), _ptr(out_sc))
    if rc:
        raise RuntimeError("oracle merge failed (%d)" % rc)
    return out_ids, out_sc


def retrieve(corpus, regions, offsets, k, K, row_scale=None, nthreads=0):
    """Whole path: (reg_ids [R,k], reg_scores [R,k], out_ids [Q,K], out_scores [Q,K])."""
    lib = _load()
    cb, ce, sc = _corpus_args(corpus, row_scale)
    c = cb if cb is not None else ce
    regions = np.ascontiguousarray(regions, dtype=np.uint16)
    offsets = np.ascontiguousarray(offsets, dtype=np.int32)
    N, d = c.shape
    R = regions.shape[0]
    Q = offsets.shape[0] - 1
    reg_ids = np.empty((R, k), dtype=np.int64)
    reg_sc = np.empty((R, k), dtype=np.float64)
    out_ids = np.empty((Q, K), dtype=np.int64)
    out_sc = np.empty((Q, K), dtype=np.float64)
    rc = lib.skip_oracle_retrieve(_ptr(cb), _ptr(ce), _ptr(sc), N, d, _ptr(regions), _ptr(offsets),
                                  Q, R, k, K, _ptr(reg_ids), _ptr(reg_sc), _ptr(out_ids),
                                  _ptr(out_sc), int(nthreads))
    if rc:
        raise RuntimeError("oracle retrieve failed (%d)" % rc)
    return reg_ids, reg_sc, out_ids, out_sc


def score_matrix(corpus, regions, row_scale=None):
    """Every s(r, i) in fp64: [R, N]."""
    lib = _load()
    cb, ce, sc = _corpus_args(corpus, row_scale)
    c = cb if cb is not None else ce
    regions = np.ascontiguousarray(regions, dtype=np.uint16)
    N, d = c.shape
    R = regions.shape[0]
    out = np.empty((R, N), dtype=np.float64)
    rc = lib.skip_oracle_score_matrix(_ptr(cb), _ptr(ce), _ptr(sc), N, d, _ptr(regions), R,
                                      _ptr(out))
    if rc:
        raise RuntimeError("oracle score_matrix failed (%d)" % rc)
    return out


def scores_at(corpus, regions, region_idx, ids, row_scale=None):
    """s(region_idx[t], ids[t]) in fp64 for each t (NaN for ids outside [0, N))."""
    lib = _load()
    cb, ce, sc = _corpus_args(corpus, row_scale)
    c = cb if cb is not None else ce
    regions = np.ascontiguousarray(regions, dtype=np.uint16)
    region_idx = np.ascontiguousarray(region_idx, dtype=np.int64).ravel()
    ids = np.ascontiguousarray(ids, dtype=np.int64).ravel()
    N, d = c.shape
    out = np.empty(ids.shape[0], dtype=np.float64)
    rc = lib.skip_oracle_scores_at(_ptr(cb), _ptr(ce), _ptr(sc), N, d, _ptr(regions),
                                   _ptr(region_idx), _ptr(ids), ids.shape[0], _ptr(out))
    if rc:
        raise RuntimeError("oracle scores_at failed (%d)" % rc)
    return out


def bf16_round(x: float) -> int:
    """x rounded to bf16 (ties to even); the bit pattern."""
    return int(_load().skip_oracle_bf16_round(float(x)))


def skv_count(n_nonempty: int, rho: float) -> int:
    """ceil(rho * |K| - 1e-3) clamped to [0, |K|]: how many gated passages are kept."""
    return int(_load().skip_oracle_skv_count(int(n_nonempty), float(rho)))


def skv(corpus, ids, qbar, vbar, w1, b1, w2, b2, tau=0.5, rho=0.6):
    """SKV gate on candidate lists (Def. B.4 and the Alg. 1 TopK).

    corpus uint16 [N, d] (bf16 bits); ids int64 [Q, K] (-1 = empty slot);
    qbar, vbar uint16 [Q, d]; w1 uint16 [H, 5d]; b1, w2 float32 [H]; b2 float.
    Returns a dict: nu_all, bound (float64 [Q, K]), ids (int64 [Q, K]),
    nu (float64 [Q, K]), count (int32 [Q]).
    """
    lib = _load()
    corpus = np.ascontiguousarray(corpus, dtype=np.uint16)
    ids = np.ascontiguousarray(ids, dtype=np.int64)
    qbar = np.ascontiguousarray(qbar, dtype=np.uint16)
    vbar = np.ascontiguousarray(vbar, dtype=np.uint16)
    w1 = np.ascontiguousarray(w1, dtype=np.uint16)
    b1 = np.ascontiguousarray(b1, dtype=np.float32)
    w2 = np.ascontiguousarray(w2, dtype=np.float32)
    N, d = corpus.shape
    Q, K = ids.shape
    H = w1.shape[0]
    if w1.shape[1] != 5 * d or qbar.shape != (Q, d) or vbar.shape != (Q, d) or b1.shape != (H,) \
            or w2.shape != (H,):
        raise ValueError("skv: inconsistent shapes")
    nu_all = np.empty((Q, K), np.float64)
    bound = np.empty((Q, K), np.float64)
    out_ids = np.empty((Q, K), np.int64)
    out_nu = np.empty((Q, K), np.float64)
    count = np.empty(Q, np.int32)
    rc = lib.skip_oracle_skv(_ptr(corpus), N, d, _ptr(ids), Q, K, _ptr(qbar), _ptr(vbar), _ptr(w1),
                             _ptr(b1), _ptr(w2), float(b2), H, float(tau), float(rho), _ptr(nu_all),
                             _ptr(bound), _ptr(out_ids), _ptr(out_nu), _ptr(count))
    if rc:
        raise RuntimeError("oracle skv failed (%d)" % rc)
    return {"nu_all": nu_all, "bound": bound, "ids": out_ids, "nu": out_nu, "count": count}


def ivf_assign(corpus, centroids):
    """list(i) = argmax_l <x_i, c_l> (ties: lower l); int32 [N]."""
    lib = _load()
    corpus = np.ascontiguousarray(corpus, dtype=np.uint16)
    centroids = np.ascontiguousarray(centroids, dtype=np.uint16)
    N, d = corpus.shape
    out = np.empty(N, np.int32)
    if lib.skip_oracle_ivf_assign(_ptr(corpus), N, d, _ptr(centroids), centroids.shape[0], _ptr(out)):
        raise RuntimeError("oracle ivf_assign failed")
    return out


def pq_encode(corpus, centroids, lists, codebook):
    """PQ codes of the residuals x_i - c_list(i): uint8 [N, M]; codebook
    float32 [M, ksub, d/M] (ties: lower codeword)."""
    lib = _load()
    corpus = np.ascontiguousarray(corpus, dtype=np.uint16)
    centroids = np.ascontiguousarray(centroids, dtype=np.uint16)
    lists = np.ascontiguousarray(lists, dtype=np.int32)
    codebook = np.ascontiguousarray(codebook, dtype=np.float32)
    N, d = corpus.shape
    M, ksub = codebook.shape[0], codebook.shape[1]
    out = np.empty((N, M), np.uint8)
    if lib.skip_oracle_pq_encode(_ptr(corpus), N, d, _ptr(centroids), _ptr(lists), _ptr(codebook), M, ksub,
                                 _ptr(out)):
        raise RuntimeError("oracle pq_encode failed")
    return out


def ivf_lists(lists, C):
    """Inverted lists: (offsets int64 [C+1], ids int64 [N] grouped by list,
    ascending within a list)."""
    lists = np.asarray(lists, np.int64)
    ids = np.argsort(lists, kind="stable").astype(np.int64)
    counts = np.bincount(lists, minlength=C)
    offsets = np.zeros(C + 1, np.int64)
    offsets[1:] = np.cumsum(counts)
    return offsets, ids


def ivfpq_build(corpus, centroids, codebook):
    """The whole index: dict(lists, codes, offsets, ids)."""
    lists = ivf_assign(corpus, centroids)
    codes = pq_encode(corpus, centroids, lists, codebook)
    offsets, ids = ivf_lists(lists, np.asarray(centroids).shape[0])
    return {"lists": lists, "codes": codes, "offsets": offsets, "ids": ids}


def ivfpq_search(index, centroids, codebook, regions, nprobe, k):
    """(ids int64 [R, k], scores float64 [R, k], probes int32 [R, nprobe])."""
    lib = _load()
    centroids = np.ascontiguousarray(centroids, dtype=np.uint16)
    codebook = np.ascontiguousarray(codebook, dtype=np.float32)
    regions = np.ascontiguousarray(regions, dtype=np.uint16)
    offsets = np.ascontiguousarray(index["offsets"], dtype=np.int64)
    ids = np.ascontiguousarray(index["ids"], dtype=np.int64)
    codes = np.ascontiguousarray(index["codes"], dtype=np.uint8)
    C, d = centroids.shape
    M, ksub = codebook.shape[0], codebook.shape[1]
    R = regions.shape[0]
    out_ids = np.empty((R, k), np.int64)
    out_sc = np.empty((R, k), np.float64)
    probes = np.empty((R, nprobe), np.int32)
    if lib.skip_oracle_ivfpq_search(_ptr(centroids), C, d, _ptr(offsets), _ptr(ids), _ptr(codes), _ptr(codebook),
                                    M, ksub, _ptr(regions), R, int(nprobe), int(k), _ptr(out_ids), _ptr(out_sc),
                                    _ptr(probes)):
        raise RuntimeError("oracle ivfpq_search failed")
    return out_ids, out_sc, probes


def ivfpq_search_refine(index, centroids, codebook, regions, nprobe, k, ks, corpus, row_scale=None):
    """IVF-PQ search followed by an exact re-rank (the usual refinement of an
    IVF-PQ shortlist): each region's best ks entries by s^ (ivfpq_search),
    re-scored with the exact fp64 inner product (scores_at), the k best by
    (score desc, id asc).  Returns (ids int64 [R, k], scores float64 [R, k])."""
    s_ids, _, _ = ivfpq_search(index, centroids, codebook, regions, nprobe, ks)
    R = s_ids.shape[0]
    out_ids = np.full((R, k), -1, np.int64)
    out_sc = np.full((R, k), -np.inf)
    for r in range(R):
        cand = s_ids[r][s_ids[r] >= 0]
        if cand.size == 0:
            continue
        ex = scores_at(corpus, regions, np.full(cand.size, r), cand, row_scale=row_scale)
        order = np.lexsort((cand, -ex))[:k]
        out_ids[r, :order.size] = cand[order]
        out_sc[r, :order.size] = ex[order]
    return out_ids, out_sc


def ivfpq_scores_at(index, centroids, codebook, regions, region_idx, ids):
    """s^(q_r, i) at chosen (region, id) pairs (NaN outside [0, N))."""
    lib = _load()
    centroids = np.ascontiguousarray(centroids, dtype=np.uint16)
    codebook = np.ascontiguousarray(codebook, dtype=np.float32)
    regions = np.ascontiguousarray(regions, dtype=np.uint16)
    lists = np.ascontiguousarray(index["lists"], dtype=np.int32)
    codes = np.ascontiguousarray(index["codes"], dtype=np.uint8)
    region_idx = np.ascontiguousarray(region_idx, dtype=np.int64).ravel()
    ids = np.ascontiguousarray(ids, dtype=np.int64).ravel()
    M, ksub = codebook.shape[0], codebook.shape[1]
    out = np.empty(ids.shape[0], np.float64)
    if lib.skip_oracle_ivfpq_scores_at(_ptr(centroids), centroids.shape[1], _ptr(lists), _ptr(codes),
                                       lists.shape[0], _ptr(codebook), M, ksub, _ptr(regions), _ptr(region_idx),
                                       _ptr(ids), ids.shape[0], _ptr(out)):
        raise RuntimeError("oracle ivfpq_scores_at failed")
    return out


def qvs_count(L: int, rho: float) -> int:
    """ceil(rho * L - 1e-3) clamped to [0, L]: tokens kept per image."""
    return int(_load().skip_oracle_qvs_count(int(L), float(rho)))


def qvs(tokens, fq, wv, bv, wb, rho):
    """QVS scores and pruning.  tokens uint16 [B, L, d] (bf16 bits); fq uint16
    [B, dk]; wv uint16 [dk, d]; bv float32 [dk] or None; wb float32 [d].
    Returns (logits float64 [B, L], idx int32 [B, n], score float64 [B, n])."""
    lib = _load()
    tokens = np.ascontiguousarray(tokens, dtype=np.uint16)
    fq = np.ascontiguousarray(fq, dtype=np.uint16)
    wv = np.ascontiguousarray(wv, dtype=np.uint16)
    wb = np.ascontiguousarray(wb, dtype=np.float32)
    bv = None if bv is None else np.ascontiguousarray(bv, dtype=np.float32)
    B, L, d = tokens.shape
    dk = wv.shape[0]
    n = qvs_count(L, rho)
    logits = np.empty((B, L), np.float64)
    idx = np.empty((B, n), np.int32)
    score = np.empty((B, n), np.float64)
    if lib.skip_oracle_qvs(_ptr(tokens), B, L, d, _ptr(fq), _ptr(wv), _ptr(bv), _ptr(wb), dk, float(rho),
                           _ptr(logits), _ptr(idx), _ptr(score)):
        raise RuntimeError("oracle qvs failed")
    return logits, idx, score


def bsca_edges_count(P: int, dbar: float) -> int:
    """ceil(dbar * P - 1e-3): edges a question keeps (before ties at tau_e)."""
    return int(_load().skip_oracle_bsca_edges_count(int(P), float(dbar)))


def bsca(vis_offsets, chunk_offsets, hv, qh, hk, kh, vh, rmax, dbar=4.0, edge_mask=None):
    """BSCA per question.  Offsets int32 [Q+1]; hv, qh uint16 (bf16 bits)
    [Nv, dp] / [Nv, dh]; hk, kh, vh uint16 [Nc, dp] / [Nc, dh] / [Nc, dout].
    Returns dict(cos float64 [Nv, rmax], tau float64 [Q], degree int32 [Nv],
    out float64 [Nv, dout]).  edge_mask (uint8 [Nv, rmax]) replaces the
    threshold rule when given."""
    lib = _load()
    vo = np.ascontiguousarray(vis_offsets, dtype=np.int32)
    co = np.ascontiguousarray(chunk_offsets, dtype=np.int32)
    hv, qh, hk, kh, vh = (np.ascontiguousarray(a, dtype=np.uint16) for a in (hv, qh, hk, kh, vh))
    Q = vo.shape[0] - 1
    Nv, dp = hv.shape
    dh, dout = qh.shape[1], vh.shape[1]
    em = None if edge_mask is None else np.ascontiguousarray(edge_mask, dtype=np.uint8)
    cos = np.empty((Nv, rmax), np.float64)
    tau = np.empty(Q, np.float64)
    deg = np.empty(Nv, np.int32)
    out = np.empty((Nv, dout), np.float64)
    if lib.skip_oracle_bsca(_ptr(vo), _ptr(co), Q, _ptr(hv), _ptr(qh), _ptr(hk), _ptr(kh), _ptr(vh), dp, dh, dout,
                            int(rmax), float(dbar), _ptr(em), _ptr(cos), _ptr(tau), _ptr(deg), _ptr(out)):
        raise RuntimeError("oracle bsca failed")
    return {"cos": cos, "tau": tau, "degree": deg, "out": out}
