"""Seeded synthetic inputs for region-conditional sparse retrieval (RCSR).

This module is shared by the CUDA path's tests and benchmark and by the CPU
oracle.  It only draws and quantises inputs: it holds no scoring, selection,
merging or deduplication arithmetic.

What the inputs stand in for (paper §4.1 "Knowledge corpora"/"Implementation",
App. I.1 "Retrieval index", App. I.4 hyperparameter table): a passage corpus
of 1.7M-109M entries with 768-dimensional index vectors (Wikipedia 6.5M,
WikiData 8.2M, the ViQuAE KB 1.7M, Wikipedia 21M + Wikidata 88M), and per
question up to 8 (main text) or more region query embeddings q_{r_i}
(App. B.2, Eq. rcsr_query).  None of those corpora or trained encoders exist
here, so rows and queries are drawn from the distributions below.

Recipe (one per workload, seeds fixed per workload):

* corpus seed = workload index, region seed = 1000 + workload index;
* ``gaussian`` rows: x ~ N(0, I_d), then x / ||x||;
* ``clustered`` rows: centres c ~ N(0, I_d) normalised; each row draws a
  centre uniformly and sets x = normalise(c + sigma * N(0, I_d)) with
  sigma = 0.3 / sqrt(d) per coordinate (noise norm ~0.3, cos(x, c) ~ 0.96);
* regions of gaussian workloads: N(0, I_d) normalised;
* regions of clustered workloads: each question picks 1..4 "entity" centres
  uniformly from the corpus centres, each of its regions picks one of them
  and applies the same noise model;
* bf16 = round-to-nearest-even of the fp32 value (``torch.bfloat16``);
* e4m3 = OCP float8_e4m3fn of x / scale_i, round-to-nearest-even, with
  scale_i = max_j |x_ij| / 448 (1.0 for an all-zero row);
* ragged region counts are U{lo..hi} per question from the region seed.

Generation is chunked (``CHUNK`` rows per draw, each chunk with its own
derived seed) so that multi-GB corpora can be drawn straight into device
memory.  The same seed gives the same bytes on the same device type and
PyTorch build; CPU- and CUDA-drawn inputs differ from each other.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import torch

CHUNK = 1 << 20  # rows per generator draw


@dataclasses.dataclass(frozen=True)
class WorkloadSpec:
    name: str
    index: int          # workload index: corpus seed, region seed = 1000 + index
    N: int              # corpus rows
    d: int              # embedding dimension
    dtype: str          # "bf16" or "e4m3"
    Q: int              # questions
    regions: tuple      # (lo, hi) regions per question, inclusive
    k_region: int       # per-region top-k' (paper: k', k_r)
    K: int              # merged top-K per question
    corpus: str         # "gaussian" or "clustered"
    centres: int = 0    # cluster count for clustered corpora

    @property
    def fixed_regions(self) -> bool:
        return self.regions[0] == self.regions[1]


# The five workloads the method is measured on: a tiny exact check, a 1M
# clustered corpus, a 10M throughput batch, a 6M fp8 latency batch and a 20M
# ragged pruned batch.
WORKLOADS = {
    "tiny_100k": WorkloadSpec("tiny_100k", 0, 100_000, 768, "bf16", 4, (8, 8), 10, 20, "gaussian"),
    "clustered_1m": WorkloadSpec("clustered_1m", 1, 1_000_000, 768, "bf16", 64, (16, 16), 20, 50,
                                 "clustered", 1024),
    "throughput_10m": WorkloadSpec("throughput_10m", 2, 10_000_000, 768, "bf16", 256, (16, 16), 20, 50,
                                   "clustered", 1024),
    "latency_fp8_6m": WorkloadSpec("latency_fp8_6m", 3, 6_000_000, 1024, "e4m3", 1, (32, 32), 10, 100,
                                   "gaussian"),
    "ragged_20m": WorkloadSpec("ragged_20m", 4, 20_000_000, 512, "bf16", 1024, (1, 32), 100, 100,
                               "clustered", 4096),
}


@dataclasses.dataclass
class Workload:
    spec: WorkloadSpec
    corpus: torch.Tensor            # [N, d] bfloat16, or uint8 holding e4m3 bytes
    row_scale: Optional[torch.Tensor]  # [N] float32 for e4m3, else None
    regions: torch.Tensor           # [R_total, d] bfloat16
    offsets: torch.Tensor           # [Q + 1] int32, offsets[0] = 0
    centres: Optional[torch.Tensor] = None  # [C, d] float32 (clustered only)

    @property
    def R_total(self) -> int:
        return int(self.regions.shape[0])


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _normalise(x: torch.Tensor) -> torch.Tensor:
    n = torch.linalg.vector_norm(x, dim=1, keepdim=True)
    return x / torch.where(n > 0, n, torch.ones_like(n))


def draw_centres(spec_or_seed, C: int, d: int, device="cpu") -> torch.Tensor:
    seed = spec_or_seed.index if isinstance(spec_or_seed, WorkloadSpec) else int(spec_or_seed)
    g = _gen(seed * 7919 + 17, device)
    return _normalise(torch.randn(C, d, generator=g, device=device, dtype=torch.float32))


def corpus_rows_fp32(seed: int, n0: int, n: int, d: int, kind: str,
                     centres: Optional[torch.Tensor], device="cpu", return_centres: bool = False):
    """fp32 unit rows [n0, n0 + n) of a corpus; n0 must be a multiple of CHUNK
    unless the whole draw lies in one chunk.  With return_centres (clustered
    corpora), also the index of the centre each row was drawn around."""
    out = torch.empty(n, d, dtype=torch.float32, device=device)
    which = torch.full((n,), -1, dtype=torch.int64, device=device)
    done = 0
    while done < n:
        row = n0 + done
        chunk = row // CHUNK
        off = row - chunk * CHUNK
        take = min(n - done, CHUNK - off)
        g = _gen(seed * 1_000_003 + chunk, device)
        if kind == "gaussian":
            x = torch.randn(off + take, d, generator=g, device=device, dtype=torch.float32)[off:]
        elif kind == "clustered":
            C = centres.shape[0]
            a = torch.randint(0, C, (off + take,), generator=g, device=device)[off:]
            z = torch.randn(off + take, d, generator=g, device=device, dtype=torch.float32)[off:]
            x = centres[a] + (0.3 / math.sqrt(d)) * z
            which[done:done + take] = a
        else:
            raise ValueError(kind)
        out[done:done + take] = _normalise(x)
        done += take
    return (out, which) if return_centres else out


def quantise_e4m3(x: torch.Tensor):
    """Per-row scaled OCP e4m3: returns (uint8 bytes [n, d], float32 scale [n])."""
    amax = x.abs().amax(dim=1)
    scale = torch.where(amax > 0, amax / 448.0, torch.ones_like(amax)).to(torch.float32)
    q = (x / scale[:, None]).clamp(-448.0, 448.0).to(torch.float8_e4m3fn)
    return q.view(torch.uint8), scale


def make_corpus(spec: WorkloadSpec, device="cpu", N: Optional[int] = None):
    """Corpus of the workload (optionally only its first N rows).
    Returns (corpus, row_scale, centres)."""
    N = spec.N if N is None else N
    centres = draw_centres(spec, spec.centres, spec.d, device) if spec.corpus == "clustered" else None
    if spec.dtype == "bf16":
        corpus = torch.empty(N, spec.d, dtype=torch.bfloat16, device=device)
        scale = None
    else:
        corpus = torch.empty(N, spec.d, dtype=torch.uint8, device=device)
        scale = torch.empty(N, dtype=torch.float32, device=device)
    for n0 in range(0, N, CHUNK):
        n = min(CHUNK, N - n0)
        x = corpus_rows_fp32(spec.index, n0, n, spec.d, spec.corpus, centres, device)
        if spec.dtype == "bf16":
            corpus[n0:n0 + n] = x.to(torch.bfloat16)
        else:
            q, s = quantise_e4m3(x)
            corpus[n0:n0 + n] = q
            scale[n0:n0 + n] = s
        del x
    return corpus, scale, centres


def region_counts(spec: WorkloadSpec, Q: Optional[int] = None) -> torch.Tensor:
    Q = spec.Q if Q is None else Q
    lo, hi = spec.regions
    if lo == hi:
        return torch.full((Q,), lo, dtype=torch.int64)
    g = _gen(1000 + spec.index, "cpu")
    return torch.randint(lo, hi + 1, (Q,), generator=g)


def offsets_from_counts(counts) -> torch.Tensor:
    counts = torch.as_tensor(counts, dtype=torch.int64)
    off = torch.zeros(counts.numel() + 1, dtype=torch.int64)
    off[1:] = torch.cumsum(counts, 0)
    return off.to(torch.int32)


def make_regions(spec: WorkloadSpec, centres: Optional[torch.Tensor], device="cpu",
                 Q: Optional[int] = None):
    """Region query batch (bf16 [R_total, d]) and offsets (int32 [Q+1], on CPU)."""
    counts = region_counts(spec, Q)
    offsets = offsets_from_counts(counts)
    R = int(offsets[-1])
    g = _gen(1000 + spec.index + 1_000_003, "cpu")
    if spec.corpus == "gaussian":
        x = _normalise(torch.randn(R, spec.d, generator=g, dtype=torch.float32))
    else:
        C = centres.shape[0]
        cen = centres.to("cpu")
        rows = []
        for q in range(counts.numel()):
            ne = int(torch.randint(1, 5, (1,), generator=g))
            ent = torch.randint(0, C, (ne,), generator=g)
            pick = ent[torch.randint(0, ne, (int(counts[q]),), generator=g)]
            z = torch.randn(int(counts[q]), spec.d, generator=g, dtype=torch.float32)
            rows.append(cen[pick] + (0.3 / math.sqrt(spec.d)) * z)
        x = _normalise(torch.cat(rows, 0)) if rows else torch.empty(0, spec.d)
    return x.to(torch.bfloat16).to(device), offsets


def make_workload(name_or_spec, device="cpu", N: Optional[int] = None,
                  Q: Optional[int] = None) -> Workload:
    spec = WORKLOADS[name_or_spec] if isinstance(name_or_spec, str) else name_or_spec
    corpus, scale, centres = make_corpus(spec, device, N)
    regions, offsets = make_regions(spec, centres, device, Q)
    return Workload(spec, corpus, scale, regions, offsets, centres)


def random_bf16(n: int, d: int, seed: int, device="cpu") -> torch.Tensor:
    """Unit-norm Gaussian rows as bf16 (small test inputs)."""
    g = _gen(seed, device)
    return _normalise(torch.randn(n, d, generator=g, device=device)).to(torch.bfloat16)


def bf16_bits(t: torch.Tensor):
    """uint16 numpy view of a bf16 tensor (host)."""
    return t.detach().to("cpu").contiguous().view(torch.int16).numpy().view("uint16")


# ---- inputs of the SKV passage gate (App. B.4 Def. B.4) --------------------
#
# The gate reads the question embedding qbar, the mean-pooled visual tokens
# vbar (both d-dimensional here), each candidate passage's embedding (its
# corpus row) and the two-layer MLP h_psi.  No trained encoder or MLP exists
# here, so they are drawn:
#
# * qbar: normalise(first region query of the question + 0.5 / sqrt(d) * z);
#   a question with no region draws a Gaussian unit vector; vbar: Gaussian
#   unit vector; seed 3000 + workload index (or the given seed);
# * W1 [H x 5d] ~ N(0, 1/5) (the five input blocks are unit-scale vectors, so
#   pre-activations are ~N(0, 1)), b1 ~ N(0, 0.1^2), w2 ~ N(0, 4/H),
#   b2 = 0.1; H = 512 (App. I.4, "SKV MLP hidden dim."); W1 stored bf16,
#   b1 and w2 fp32; seed 4000 + workload index;
# * standalone candidate lists: per question distinct ids in random order,
#   the last `empty` slots -1 (seeded).

SKV_HIDDEN = 512


def make_skv_mlp(d: int, hidden: int = SKV_HIDDEN, seed: int = 4000, device="cpu"):
    """(w1 bf16 [H, 5d], b1 fp32 [H], w2 fp32 [H], b2 float)."""
    g = _gen(seed, "cpu")
    w1 = (torch.randn(hidden, 5 * d, generator=g) / math.sqrt(5.0)).to(torch.bfloat16)
    b1 = 0.1 * torch.randn(hidden, generator=g)
    w2 = (2.0 / math.sqrt(hidden)) * torch.randn(hidden, generator=g)
    return w1.to(device), b1.to(device), w2.to(device), 0.1


def make_skv_queries(regions: torch.Tensor, offsets, seed: int = 3000, device="cpu"):
    """(qbar bf16 [Q, d], vbar bf16 [Q, d]) for a region batch."""
    offsets = torch.as_tensor(offsets).to("cpu")
    Q = offsets.numel() - 1
    d = regions.shape[1]
    g = _gen(seed, "cpu")
    reg = regions.to("cpu").float()
    z = torch.randn(Q, d, generator=g)
    lead = _normalise(torch.randn(Q, d, generator=g))
    for q in range(Q):
        if int(offsets[q + 1]) > int(offsets[q]):
            lead[q] = reg[int(offsets[q])]
    qbar = _normalise(lead + (0.5 / math.sqrt(d)) * z)
    vbar = _normalise(torch.randn(Q, d, generator=g))
    return qbar.to(torch.bfloat16).to(device), vbar.to(torch.bfloat16).to(device)


def make_candidate_ids(N: int, Q: int, K: int, empty, seed: int) -> torch.Tensor:
    """int64 [Q, K]: distinct ids per question, the last empty[q] slots -1."""
    g = _gen(seed, "cpu")
    out = torch.full((Q, K), -1, dtype=torch.int64)
    empty = torch.as_tensor(empty).expand(Q) if not torch.is_tensor(empty) or empty.dim() == 0 \
        else torch.as_tensor(empty)
    for q in range(Q):
        n = K - int(empty[q])
        if n > 0:
            out[q, :n] = torch.randperm(N, generator=g)[:n]
    return out



# ---- inputs of the IVF-PQ variant ----------------------------------------
#
# The paper's index (FAISS IVF-PQ, 1,024 or 4,096 centroids, PQ64) was
# trained on its corpus; no trained index exists here.  For the clustered
# workloads the IVF centroids are the generator's own centres (1,024 for the
# 1M and 10M corpora, 4,096 for the 20M one), as bf16.  The PQ codebook is
# sample-based: codeword j of sub-space m is sub-vector m of the residual
# bf16(x_i) - bf16(c_{a_i}) of corpus row i = m * ksub + j, where a_i is the
# centre the generator drew row i around (no k-means refinement).

def make_ivf_centroids(spec: WorkloadSpec, device="cpu") -> torch.Tensor:
    """bf16 [C, d]: the clustered corpus's centres."""
    if spec.corpus != "clustered":
        raise ValueError("IVF centroids are drawn for clustered corpora")
    return draw_centres(spec, spec.centres, spec.d, device).to(torch.bfloat16)


def make_pq_codebook(spec: WorkloadSpec, M: int, ksub: int = 256, device="cpu") -> torch.Tensor:
    """float32 [M, ksub, d / M] sample-based PQ codebook (see above)."""
    if spec.d % M:
        raise ValueError("M must divide d")
    centres = draw_centres(spec, spec.centres, spec.d, "cpu")
    n = M * ksub
    x, a = corpus_rows_fp32(spec.index, 0, n, spec.d, spec.corpus, centres, "cpu", return_centres=True)
    r = x.to(torch.bfloat16).float() - centres[a].to(torch.bfloat16).float()
    ds = spec.d // M
    cb = torch.empty(M, ksub, ds)
    for m in range(M):
        cb[m] = r[m * ksub:(m + 1) * ksub, m * ds:(m + 1) * ds]
    return cb.to(device)


def train_pq_codebook(spec: WorkloadSpec, M: int, ksub: int = 256, sample: int = 65536, iters: int = 12,
                      device="cpu") -> torch.Tensor:
    """float32 [M, ksub, d / M] PQ codebook trained by k-means (Lloyd's
    algorithm, squared L2) on the residuals bf16(x_i) - bf16(c_{a_i}) of the
    first `sample` corpus rows, each sub-space on its own; it starts from the
    sample-based codebook above, and a codeword that loses all its points
    keeps its place.  Index training, like the paper's FAISS index (trained
    offline on its corpus), is input preparation here: the library and the
    oracle both take the codebook as given."""
    if spec.d % M:
        raise ValueError("M must divide d")
    centres = draw_centres(spec, spec.centres, spec.d, "cpu")
    x, a = corpus_rows_fp32(spec.index, 0, min(sample, spec.N), spec.d, spec.corpus, centres, "cpu",
                            return_centres=True)
    r = (x.to(torch.bfloat16).float() - centres[a].to(torch.bfloat16).float()).to(device)
    ds = spec.d // M
    sub = r.view(r.shape[0], M, ds).permute(1, 0, 2).contiguous()      # [M, n, ds]
    cb = make_pq_codebook(spec, M, ksub, device=device).clone()          # [M, ksub, ds]
    for _ in range(iters):
        # nearest codeword of every sub-vector: argmin ||r||^2 - 2 r.c + ||c||^2
        d2 = (cb * cb).sum(-1)[:, None, :] - 2.0 * torch.bmm(sub, cb.transpose(1, 2))
        assign = d2.argmin(-1)                                           # [M, n]
        sums = torch.zeros_like(cb).scatter_add_(1, assign[..., None].expand(-1, -1, ds), sub)
        cnt = torch.zeros(M, ksub, device=sub.device).scatter_add_(1, assign, torch.ones_like(assign,
                                                                                              dtype=torch.float32))
        upd = cnt > 0
        cb[upd] = sums[upd] / cnt[upd][:, None]
    return cb.to(device)


# ---- inputs of QVS (App. B.1 Def. B.1) -------------------------------------
#
# QVS scores L visual tokens per image against the question: L = 576 (a 24 x
# 24 patch grid, §4.1 / App. I.4: CLIP ViT-L/14 at 336 px), token width
# d = 1024, d_k = d (Def. B.1 maps both to R^d).  No vision encoder or trained
# QVS head exists here: tokens are Gaussian unit vectors, of which about 22%
# ("entity" patches; the paper finds ~78% background) are pulled towards an
# image direction g_b (x = normalise(z + 2 g_b)); f_q(Q) is normalise(g_b +
# N(0, I)) scaled by sqrt(d); W_v = I + N(0, 0.25/d) (so that f_v roughly
# keeps the token and entity patches score high), b_v ~ N(0, 0.01^2),
# w_b ~ N(0, 1/d).  Tokens, f_q and W_v are bf16; b_v and w_b fp32.

QVS_L, QVS_D = 576, 1024


def make_qvs_inputs(B: int, L: int = QVS_L, d: int = QVS_D, seed: int = 5000, device="cpu"):
    """(tokens bf16 [B, L, d], fq bf16 [B, d], wv bf16 [d, d], bv fp32 [d], wb fp32 [d])."""
    g = _gen(seed, "cpu")
    gdir = _normalise(torch.randn(B, d, generator=g))
    tokens = torch.empty(B, L, d, dtype=torch.bfloat16)
    for b in range(B):
        z = torch.randn(L, d, generator=g) / math.sqrt(d)
        ent = torch.rand(L, generator=g) < 0.22
        z[ent] += 2.0 * gdir[b]
        tokens[b] = _normalise(z).to(torch.bfloat16)
    fq = (math.sqrt(d) * _normalise(gdir + torch.randn(B, d, generator=g) / math.sqrt(d))).to(torch.bfloat16)
    wv = (torch.eye(d) + 0.5 * torch.randn(d, d, generator=g) / math.sqrt(d)).to(torch.bfloat16)
    bv = 0.01 * torch.randn(d, generator=g)
    wb = torch.randn(d, generator=g) / math.sqrt(d)
    return tokens.to(device), fq.to(device), wv.to(device), bv.to(device), wb.to(device)


# ---- inputs of BSCA (App. B.3 Def. B.3) ------------------------------------
#
# BSCA fuses each question's retained visual tokens (P = ceil(rho_v L): 231
# for rho_v = 0.4) with its verified chunks (R, ragged: what the SKV gate
# keeps, 16..32 here) through projections h_v, h_k (width d_p), W_Q, W_K
# (width d_h = 128, App. I.4) and W_V (width d_o).  The projected vectors are
# the inputs here: Gaussian rows (unit norm for h_v / h_k, N(0, 1) entries
# for the others), bf16; chunk counts U{16..32} per question (seeded).

def make_bsca_inputs(Q: int, P: int, R_lo: int = 16, R_hi: int = 32, dp: int = 128, dh: int = 128,
                     dout: int = 1024, seed: int = 6000, device="cpu"):
    """dict(vis_offsets, chunk_offsets (int32 [Q+1]), hv [Nv, dp], qh [Nv, dh],
    hk [Nc, dp], kh [Nc, dh], vh [Nc, dout] (bf16))."""
    g = _gen(seed, "cpu")
    counts_r = torch.randint(R_lo, R_hi + 1, (Q,), generator=g)
    vo = offsets_from_counts(torch.full((Q,), P, dtype=torch.int64))
    co = offsets_from_counts(counts_r)
    Nv, Nc = int(vo[-1]), int(co[-1])
    hv = _normalise(torch.randn(Nv, dp, generator=g))
    hk = _normalise(torch.randn(Nc, dp, generator=g))
    qh = torch.randn(Nv, dh, generator=g)
    kh = torch.randn(Nc, dh, generator=g)
    vh = torch.randn(Nc, dout, generator=g)
    bf = lambda t: t.to(torch.bfloat16).to(device)
    return {"vis_offsets": vo, "chunk_offsets": co, "hv": bf(hv), "qh": bf(qh), "hk": bf(hk), "kh": bf(kh),
            "vh": bf(vh)}
