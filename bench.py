#!/usr/bin/env python
"""Throughput of region-conditional sparse retrieval on GB300.

A step is one call of the whole path (per-region MIPS top-k over the corpus,
cross-partition merge, per-question dedup and top-K; paper §3.3 Eq. rcsr,
App. B.2 Def. B.2, Alg. 1) on one batch of questions whose region embeddings
and corpus are already resident in HBM.  The default workload is the largest
single-GPU one, the ragged pruned batch (N = 20,000,000 x d = 512 bf16 with
4,096 clusters, 1,024 questions with U{1..32} regions each, k_region = 100,
K = 100); --workload picks another.  Every corpus is larger than L2
(129 MB), so each step streams it from HBM without an explicit flush.

Printed as one JSON line: questions/s (``value``), corpus GB/s, region rows/s,
TFLOP/s, the roofline of the dominant kernel (CUDA events on the launching
stream, recorded by the library around each kernel), clocks sampled during the
timed region, the end-to-end rate through the host-buffer entry point
(host->device copies and result read-back inside the timed region), and the
CPU oracle timed on a bounded sample of the same workload.

Multi-GPU (torchrun): each rank holds a replica of the corpus and serves its
own batch of questions (weak scaling); ranks exchange nothing on the data
path, only the barrier and the max of the timings.

``--impl reference`` times the CPU oracle instead (rank 0 only), one question
per step over a prefix of the corpus, scaled to full-corpus questions/s.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "retrieval queries/s and corpus GB/s (1 GB300) as fraction of roofline"
SCORE_KERNELS = ("score_topk_tc", "score_topk_tc_e4m3", "score_topk_latency", "score_topk_latency_e4m3",
                 "score_topk_warpdot")
KERNEL_SOURCES = {
    "score_topk_tc": ["paper_2607_25422_gb300/csrc/k_tc.cu", "paper_2607_25422_gb300/csrc/tc_common.cuh",
                      "paper_2607_25422_gb300/csrc/skip_device.cuh"],
    "score_topk_tc_e4m3": ["paper_2607_25422_gb300/csrc/k_tc_fp8.cu", "paper_2607_25422_gb300/csrc/tc_common.cuh",
                           "paper_2607_25422_gb300/csrc/skip_device.cuh"],
    "score_topk_latency": ["paper_2607_25422_gb300/csrc/k_latency.cu", "paper_2607_25422_gb300/csrc/tc_common.cuh",
                           "paper_2607_25422_gb300/csrc/skip_device.cuh"],
    "score_topk_latency_e4m3": ["paper_2607_25422_gb300/csrc/k_latency.cu",
                                "paper_2607_25422_gb300/csrc/tc_common.cuh",
                                "paper_2607_25422_gb300/csrc/skip_device.cuh"],
    "score_topk_warpdot": ["paper_2607_25422_gb300/csrc/k_warpdot.cu",
                           "paper_2607_25422_gb300/csrc/skip_device.cuh"],
}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            m = json.load(f)
        return {"hbm_gbs": m["hbm_gbs"], "bf16_tflops": m["bf16_tflops"],
                "bf16_tflops_sustained": m.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def source_sha(kernel):
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES.get(kernel, []):
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel, workload):
    """DRAM bytes per launch from a committed ncu summary, if it was taken
    on the kernel as it is now."""
    p = os.path.join(ROOT, "profiles", "%s_%s.json" % (kernel, workload))
    if not os.path.exists(p):
        return None
    with open(p) as f:
        s = json.load(f)
    if s.get("source_sha") != source_sha(kernel):
        return None
    return s.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 100 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"samples": 0}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def workload_config(spec, R_total, world):
    lo, hi = spec.regions
    return {
        "workload": spec.name, "N": spec.N, "d": spec.d, "corpus_dtype": spec.dtype,
        "questions_per_gpu": spec.Q, "regions_per_question": lo if lo == hi else "U{%d..%d}" % (lo, hi),
        "R_total_per_gpu": R_total, "k_region": spec.k_region, "K": spec.K, "corpus": spec.corpus,
        "l2": "inputs larger than L2 (corpus %.2f GB > 129 MB), no flush" % (
            spec.N * spec.d * (2 if spec.dtype == "bf16" else 1) / 1e9),
        "parallelism": "replicas: corpus copy per GPU, question batches sharded across %d rank(s)" % world,
    }


def make_inputs(spec, rank, world, device):
    corpus, scale, centres = synth.make_corpus(spec, device=device)
    regions_all, offsets_all = synth.make_regions(spec, centres, "cpu", Q=spec.Q * world)
    r0, r1 = int(offsets_all[rank * spec.Q]), int(offsets_all[(rank + 1) * spec.Q])
    regions = regions_all[r0:r1].contiguous()
    offsets = (offsets_all[rank * spec.Q:(rank + 1) * spec.Q + 1] - r0).to(torch.int32)
    return corpus, scale, regions, offsets


def host_corpus(corpus, scale):
    if corpus.dtype == torch.bfloat16:
        return synth.bf16_bits(corpus), None
    return corpus.cpu().numpy(), scale.cpu().numpy()


def cpu_model():
    """The host CPU's model name (x86: 'model name'; Arm: implementer and
    part numbers), for the baseline's record."""
    try:
        with open("/proc/cpuinfo") as f:
            info = f.read()
    except OSError:
        return platform.machine()
    for key in ("model name", "Model name"):
        for line in info.splitlines():
            if line.startswith(key):
                return line.split(":", 1)[1].strip()
    fields = {}
    for line in info.splitlines():
        if ":" in line:
            k, v = line.split(":", 1)
            fields.setdefault(k.strip(), v.strip())
    parts = {"0xd0c": "Neoverse N1", "0xd40": "Neoverse V1", "0xd49": "Neoverse N2", "0xd4f": "Neoverse V2"}
    part = fields.get("CPU part", "?")
    return "%s %s (CPU implementer %s, part %s)" % (platform.machine(), parts.get(part, ""),
                                                   fields.get("CPU implementer", "?"), part)


def dedup_rate(skip, c, reg_d, offsets, k):
    """Share of the pooled region-list entries of a question that repeat an
    id already in the pool, over the batch (the paper reports 40-60% on real
    questions): one untimed skip_retrieve_regions call."""
    rid, _ = skip.skip_retrieve_regions(c, reg_d, k)
    rid = rid.cpu()
    off = offsets.numpy()
    pooled = dup = 0
    for q in range(off.size - 1):
        ids = rid[off[q]:off[q + 1]].reshape(-1)
        ids = ids[ids >= 0]
        pooled += ids.numel()
        dup += ids.numel() - torch.unique(ids).numel()
    return dup / max(1, pooled)


def cpu_baseline(spec, corpus_np, scale_np, regions, offsets, questions):
    """The oracle on a bounded sample of the batch over the full corpus.
    Ragged batches: a question with the fewest and one with the most regions
    (their mean region count is the batch's expected one); fixed batches:
    the first `questions` questions.  Scaled to questions/s of the batch,
    which extrapolates from the sample."""
    import oracle
    nthreads = len(os.sched_getaffinity(0))
    off_all = offsets.numpy().astype(np.int64)
    counts = np.diff(off_all)
    if spec.fixed_regions:
        qs = list(range(min(questions, counts.size)))
        how = "first %d questions" % len(qs)
    else:
        qs = sorted({int(np.argmin(counts)), int(np.argmax(counts))})
        how = "the questions with the fewest (%d) and the most (%d) regions" % (counts.min(), counts.max())
    rows = [r for q in qs for r in range(off_all[q], off_all[q + 1])]
    reg = synth.bf16_bits(regions[rows])
    off = np.concatenate([[0], np.cumsum(counts[qs])]).astype(np.int32)
    oracle.build()
    t0 = time.perf_counter()
    oracle.retrieve(corpus_np, reg, off, spec.k_region, spec.K, row_scale=scale_np, nthreads=nthreads)
    dt = time.perf_counter() - t0
    per_region = dt / max(1, len(rows))
    batch_s = per_region * int(off_all[-1])
    return {"value": (counts.size / batch_s) if not spec.fixed_regions else len(qs) / dt, "unit": "queries/s",
            "cores": nthreads, "kind": "oracle", "cpu": cpu_model(),
            "sample": "%s (%d regions) over the full %d-row corpus, fp64, %d OpenMP threads, %.1f s; %s" % (
                how, len(rows), spec.N, nthreads, dt,
                "scaled per region to the batch's %d regions (extrapolated)" % int(off_all[-1])
                if not spec.fixed_regions else "measured on the sample")}


def run_reference(args, spec):
    """The CPU oracle as the reference arm: one question per step over the
    first n_s corpus rows, scaled by N / n_s to full-corpus questions/s."""
    import oracle
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    oracle.build()
    nthreads = len(os.sched_getaffinity(0))
    corpus, scale, centres = synth.make_corpus(spec, device="cpu", N=min(spec.N, 1 << 18))
    regions, offsets = synth.make_regions(spec, centres, "cpu")
    cnp, snp = host_corpus(corpus, scale)
    q_regions = [synth.bf16_bits(regions[int(offsets[q]):int(offsets[q + 1])]) for q in range(spec.Q)]

    def step(i, n_s):
        reg = q_regions[i % spec.Q]
        off = np.array([0, reg.shape[0]], np.int32)
        oracle.retrieve(cnp[:n_s], reg, off, spec.k_region, spec.K,
                        row_scale=None if snp is None else snp[:n_s], nthreads=nthreads)

    n_s = cnp.shape[0]
    t0 = time.perf_counter()
    step(0, n_s)
    t_one = time.perf_counter() - t0
    budget = 120.0
    n_s = int(max(4096, min(n_s, n_s * budget / max(1e-9, t_one * (args.steps + args.warmup)))))
    for i in range(args.warmup):
        step(i, n_s)
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(i, n_s)
    dt = time.perf_counter() - t0
    value = args.steps * (n_s / spec.N) / dt
    sample = ("one question per step (%s regions) over the first %d of %d corpus rows, fp64, %d OpenMP "
              "threads; scaled by N / %d" % (spec.regions[0], n_s, spec.N, nthreads, n_s))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "queries/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(spec, int(offsets[-1]), 1),
            "cpu_baseline": {"value": value, "unit": "queries/s", "cores": nthreads, "kind": "oracle",
                             "cpu": cpu_model(), "sample": sample},
            "e2e": {"value": value, "unit": "queries/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def ivfpq_report(args, spec, skip, c, ix, cent, reg_d, off_d, kernels, build_s, peaks, ms):
    """Figures of the IVF-PQ step: recall against the exact path, the codes
    the scan reads (probed list sizes from the index offsets), the scan
    kernel's bandwidth against the HBM peak."""
    k = spec.k_region
    ivf_ids, _ = skip.skip_ivfpq_search_regions(ix, reg_d, args.nprobe, k)
    ex_ids, _ = skip.skip_retrieve_regions(c, reg_d, k)
    q_ivf, _ = skip.skip_ivfpq_search(ix, reg_d, off_d, args.nprobe, k, spec.K)
    q_ex, _ = skip.skip_retrieve(c, reg_d, off_d, k, spec.K)
    torch.cuda.synchronize()

    def recall(a, b, n):
        a, b = a.cpu().numpy(), b.cpu().numpy()
        return float(np.mean([len(set(x[x >= 0]) & set(y[y >= 0])) / max(1, min(n, (y >= 0).sum()))
                              for x, y in zip(a, b)]))

    # recall and step time over a sweep of probes (after the timed region)
    sweep = {}
    for npb in (8, 32, 128):
        if npb > int(cent.shape[0]):
            continue
        out_i = torch.empty_like(q_ivf)
        out_s = torch.empty(q_ivf.shape, dtype=torch.float32, device=q_ivf.device)
        for _ in range(3):
            skip.skip_ivfpq_search(ix, reg_d, off_d, npb, k, spec.K, out_i, out_s)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(10):
            skip.skip_ivfpq_search(ix, reg_d, off_d, npb, k, spec.K, out_i, out_s)
        e1.record()
        torch.cuda.synchronize()
        r_ids, _ = skip.skip_ivfpq_search_regions(ix, reg_d, npb, k)
        sweep[npb] = {"recall_region_at_k": recall(r_ids, ex_ids, k), "recall_question_at_K": recall(out_i, q_ex, spec.K),
                      "ms_per_step": e0.elapsed_time(e1) / 10}
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    skip.skip_retrieve(c, reg_d, off_d, k, spec.K)
    e0.record()
    for _ in range(5):
        skip.skip_retrieve(c, reg_d, off_d, k, spec.K)
    e1.record()
    torch.cuda.synchronize()
    exact_ms = e0.elapsed_time(e1) / 5
    off, _, _ = skip.skip_ivfpq_lists(ix)
    sizes = (off[1:] - off[:-1]).double()
    probes = torch.topk(reg_d.float() @ cent.float().T, args.nprobe, dim=1).indices
    scanned = float(sizes[probes].sum())
    scan = kernels.get("ivfpq_scan", {"ms": float("nan"), "launches": 1})
    scan_ms = scan["ms"] / max(1, scan["launches"])
    code_bytes = scanned * (args.pq_m + 4)
    return {
        "ivfpq": {"C": int(cent.shape[0]), "M": args.pq_m, "nprobe": args.nprobe, "build_s": build_s,
                  "codebook": "k-means on 65,536 rows' residuals" if args.pq_train else "sample-based",
                  "refine": args.ivf_refine,
                  "nprobe_sweep": sweep,
                  "recall_region_at_k": recall(ivf_ids, ex_ids, k), "recall_question_at_K": recall(q_ivf, q_ex, spec.K),
                  "codes_scanned_per_step": scanned, "scan_kernel_ms": scan_ms,
                  "scan_gbs": code_bytes / (scan_ms / 1e3) / 1e9,
                  "scan_frac_of_hbm": code_bytes / (scan_ms / 1e3) / 1e9 / peaks["hbm_gbs"],
                  "exact_step_ms_for_reference": exact_ms,
                  "index_bytes": spec.N * (args.pq_m + 4),
                  "note": "codes of probed lists mostly served from L2 when the index fits in 129 MB"},
        "roofline": {"bound": "hbm", "achieved": code_bytes / (scan_ms / 1e3) / 1e9, "peak": peaks["hbm_gbs"],
                     "unit": "GB/s", "frac": code_bytes / (scan_ms / 1e3) / 1e9 / peaks["hbm_gbs"], "traffic": None,
                     "kernel": "ivfpq_scan", "kernel_ms": scan_ms, "algorithmic_bytes_per_launch": code_bytes,
                     "peak_source": peaks["source"]},
    }



def timed_steps_flushed(step, steps, stream, dev):
    """Device time of `steps` calls of step(), each bracketed by its own CUDA
    events on `stream`, with L2 flushed between them (a 256 MB buffer larger
    than the 129 MB L2 is rewritten outside the events), for inputs that would
    otherwise stay in L2.  Returns (total ms, last output)."""
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    out = None
    with torch.cuda.stream(stream):
        for a, b in evs:
            flush.fill_(1)
            a.record(stream)
            out = step()
            b.record(stream)
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in evs), out

def run_bsca(args, spec, skip):
    """BSCA bench: one question per workload question (Q), 231 retained visual
    tokens (rho_v = 0.4 of 576), 16..32 verified chunks, d_p = d_h = 128,
    d_o = 1024, mean degree --dbar.  Bound by the fp32 output it writes."""
    world, rank, local = dist_setup()
    dev = torch.device("cuda", torch.cuda.current_device())
    Q, P, dp, dh, dout = spec.Q, 231, 128, 128, 1024
    x = synth.make_bsca_inputs(Q, P, 16, 32, dp, dh, dout)
    Nv, Nc = int(x["vis_offsets"][-1]), int(x["chunk_offsets"][-1])
    xd = {k: v.to(dev).contiguous() for k, v in x.items()}
    h = skip.skip_bsca_create(dp, dh, dout, Q, Nv)
    stream = torch.cuda.current_stream()

    def step():
        return skip.skip_bsca_run(h, xd["vis_offsets"], xd["chunk_offsets"], xd["hv"], xd["qh"], xd["hk"], xd["kh"],
                                  xd["vh"], args.dbar, stream=stream)
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    sampler = ClockSampler(torch.cuda.current_device())
    barrier(world)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.3)
    t_ms, out = timed_steps_flushed(step, args.steps, stream, dev)
    clocks = sampler.stop()
    ms = max_over_ranks(t_ms, world)
    if skip.skip_bsca_sync_status(h) != skip.SKIP_OK:
        raise SystemExit("bsca kernel status")
    # end to end: host projections in, the fused tokens out
    xh = {k: v.pin_memory() for k, v in x.items()}
    out_h = torch.empty(Nv, dout, dtype=torch.float32).pin_memory()

    def e2e_step():
        for k in xd:
            xd[k].copy_(xh[k], non_blocking=True)
        o = step()
        out_h.copy_(o, non_blocking=True)
        stream.synchronize()
    for _ in range(3):
        e2e_step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        e2e_step()
    e2e_s = max_over_ranks(time.perf_counter() - t0, world)
    peaks = load_peaks()
    step_ms = ms / args.steps
    in_bytes = Nv * (dp + dh) * 2 + Nc * (dp + dh + dout) * 2
    step_bytes = in_bytes + Nv * dout * 4 + 2 * Nv * 64 * 4
    achieved = step_bytes / (step_ms / 1e3) / 1e9
    line = {
        "metric": "BSCA questions/s (sparse visual-chunk fusion) [next row]",
        "value": Q * world * args.steps / (ms / 1e3), "unit": "questions/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16 in, fp32 out", "data": "synthetic",
        "config": {"workload": "bsca_%dq_%dtok" % (Q, P), "questions_per_gpu": Q, "visual_tokens": P,
                   "chunks": "U{16..32}", "d_p": dp, "d_h": dh, "d_o": dout, "dbar": args.dbar,
                   "l2": "L2 flushed between timed steps (256 MB write outside the events); "
                         "output %.1f MB written per step" % (Nv * dout * 4 / 1e6)},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": achieved / peaks["hbm_gbs"], "traffic": None, "kernel": "bsca step (3 kernels)",
                     "algorithmic_bytes_per_step": step_bytes, "peak_source": peaks["source"]},
        "clocks": clocks,
        "e2e": {"value": Q * world * args.steps / e2e_s, "unit": "questions/s", "h2d_bytes_per_step": in_bytes,
                "d2h_bytes_per_step": Nv * dout * 4, "entry_point": "skip_bsca_run with pinned host copies"},
        "gpu_launches": 3 * args.steps,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        nq = 4
        sub = synth.make_bsca_inputs(nq, P, 16, 32, dp, dh, dout)
        b = synth.bf16_bits
        t0 = time.perf_counter()
        oracle.bsca(sub["vis_offsets"], sub["chunk_offsets"], b(sub["hv"]), b(sub["qh"]), b(sub["hk"]), b(sub["kh"]),
                    b(sub["vh"]), 64, args.dbar)
        dt = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": nq / dt, "unit": "questions/s", "cores": 1, "kind": "oracle",
                                "sample": "%d questions of the same shape (fp64, one thread)" % nq}
    h.free()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_qvs(args, spec, skip):
    """QVS bench: one image per question of the workload (B = Q), L = 576
    tokens of d = 1024, d_k = d, rho_v from --rho-v; HBM-bound token scan."""
    world, rank, local = dist_setup()
    dev = torch.device("cuda", torch.cuda.current_device())
    B = spec.Q
    L, d = synth.QVS_L, synth.QVS_D
    tokens, fq, wv, bv, wb = synth.make_qvs_inputs(B, L, d)
    head = skip.skip_qvs_create(wv.to(dev), bv.to(dev), wb.to(dev), B, L)
    tok_d, fq_d = tokens.to(dev), fq.to(dev)
    n = skip.skip_qvs_count(L, args.rho_v)
    idx = torch.empty(B, n, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()

    def step():
        return skip.skip_qvs_prune(head, tok_d, fq_d, args.rho_v, with_tokens=True, stream=stream)
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    # per-kernel times: one profiled pass of events around each launch is not
    # available without a handle, so the scan kernel's share comes from ncu;
    # the step time here is the whole prune.
    sampler = ClockSampler(torch.cuda.current_device())
    barrier(world)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.3)
    t_ms, _ = timed_steps_flushed(step, args.steps, stream, dev)
    clocks = sampler.stop()
    ms = max_over_ranks(t_ms, world)
    # end to end: host tokens in, kept indices and scores out
    tok_h, fq_h = tokens.pin_memory(), fq.pin_memory()
    idx_h = torch.empty(B, n, dtype=torch.int32).pin_memory()
    sc_h = torch.empty(B, n, dtype=torch.float32).pin_memory()

    def e2e_step():
        tok_d.copy_(tok_h, non_blocking=True)
        fq_d.copy_(fq_h, non_blocking=True)
        i, sc, _ = step()
        idx_h.copy_(i, non_blocking=True)
        sc_h.copy_(sc, non_blocking=True)
        stream.synchronize()
    for _ in range(3):
        e2e_step()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        e2e_step()
    e2e_s = max_over_ranks(time.perf_counter() - t0, world)
    peaks = load_peaks()
    step_ms = ms / args.steps
    tok_bytes = B * L * d * 2
    step_bytes = tok_bytes + B * n * d * 2 + wv.numel() * 2 + B * L * 4 * 2
    achieved = step_bytes / (step_ms / 1e3) / 1e9
    line = {
        "metric": "QVS images/s (visual token pruning) [next row]", "value": B * world * args.steps / (ms / 1e3),
        "unit": "images/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": "qvs_%dx%dx%d" % (B, L, d), "images_per_gpu": B, "tokens": L, "d": d, "d_k": d,
                   "rho_v": args.rho_v, "kept": n,
                   "l2": "L2 flushed between timed steps (256 MB write outside the events); tokens %.1f MB"
                         % (tok_bytes / 1e6)},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": achieved / peaks["hbm_gbs"], "traffic": None, "kernel": "qvs step (3 kernels: split-K projected-query GEMM, logits, rank + gather)",
                     "algorithmic_bytes_per_step": step_bytes, "peak_source": peaks["source"]},
        "clocks": clocks,
        "e2e": {"value": B * world * args.steps / e2e_s, "unit": "images/s",
                "h2d_bytes_per_step": tok_bytes + B * d * 2, "d2h_bytes_per_step": B * n * 8,
                "entry_point": "skip_qvs_prune with pinned host copies in and out"},
        "gpu_launches": 3 * args.steps,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        nb = 2
        t0 = time.perf_counter()
        oracle.qvs(synth.bf16_bits(tokens[:nb]), synth.bf16_bits(fq[:nb]), synth.bf16_bits(wv), bv.numpy(),
                   wb.numpy(), args.rho_v)
        dt = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": nb / dt, "unit": "images/s", "cores": oracle.threads(), "kind": "oracle",
                                "sample": "%d images of the batch (fp64, W_v v per token as defined)" % nb}
    head.free()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", default="ragged_20m", choices=sorted(synth.WORKLOADS))
    ap.add_argument("--cpu-questions", type=int, default=8, help="questions in the oracle sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--path", default="auto", choices=["auto", "tensor", "warp", "latency"])
    ap.add_argument("--rows", type=int, default=0,
                    help="use only the first ROWS corpus rows (smaller profiling captures; not a bench line)")
    ap.add_argument("--ivfpq", action="store_true",
                    help="step = IVF-PQ search (generator centres as IVF centroids, sample-based PQ codebook)")
    ap.add_argument("--nprobe", type=int, default=32)
    ap.add_argument("--pq-m", type=int, default=64, help="PQ sub-spaces (codes of M bytes)")
    ap.add_argument("--ivf-refine", type=int, default=0,
                    help="IVF-PQ: re-rank the best r * k_region entries by s^ exactly (0: plain IVF-PQ)")
    ap.add_argument("--pq-train", action="store_true",
                    help="PQ codebook trained by k-means on 65,536 corpus rows' residuals (else sample-based)")
    ap.add_argument("--qvs", action="store_true",
                    help="step = QVS token pruning of one image per question of the workload (576 x 1024 tokens)")
    ap.add_argument("--rho-v", type=float, default=0.4)
    ap.add_argument("--bsca", action="store_true",
                    help="step = BSCA of one question per workload question: 231 visual tokens x 16..32 chunks")
    ap.add_argument("--dbar", type=float, default=4.0)
    ap.add_argument("--skv", action="store_true",
                    help="step = retrieval + SKV passage gate (skip_retrieve_skv), H = 512, tau 0.5, rho 0.6")
    ap.add_argument("--wait-timeout-ns", type=int, default=0,
                    help="cap on each in-kernel wait (0: the library's 2 s); profilers that replay a kernel "
                         "many times slow it down enough to need more")
    ap.add_argument("--resident", default="auto", choices=["auto", "never", "force"],
                    help="query blocks resident in shared memory (pair kernel, d <= 512): the library's rule, "
                         "never, or whenever the shape allows (smaller profiling captures of the same kernel)")
    ap.add_argument("--mma", default="auto", choices=["auto", "single", "pair"],
                    help="tensor-path MMA shape (auto = library's choice)")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("at least 3 warm-up steps")
    spec = synth.WORKLOADS[args.workload]
    if args.rows:
        import dataclasses
        spec = dataclasses.replace(spec, N=min(spec.N, args.rows), name="%s_rows%d" % (spec.name, args.rows))
    if args.impl == "reference":
        run_reference(args, spec)
        return

    import paper_2607_25422_gb300 as skip

    if args.qvs:
        run_qvs(args, spec, skip)
        return
    if args.bsca:
        run_bsca(args, spec, skip)
        return
    world, rank, local = dist_setup()
    dev = torch.device("cuda", torch.cuda.current_device())
    corpus, scale, regions, offsets = make_inputs(spec, rank, world, dev)
    R = regions.shape[0]
    Q = offsets.numel() - 1
    c = skip.skip_corpus_load(corpus, row_scale=scale)
    keep_host = rank == 0 and world == 1 and not args.no_cpu_baseline and not args.ivfpq
    corpus_np, scale_np = host_corpus(corpus, scale) if keep_host else (None, None)
    del corpus
    torch.cuda.empty_cache()
    c.set_option(skip.SKIP_OPT_PATH, {"auto": 0, "tensor": 1, "warp": 2, "latency": 3}[args.path])
    c.set_option(skip.SKIP_OPT_MMA, {"auto": 0, "single": 1, "pair": 2}[args.mma])
    c.set_option(skip.SKIP_OPT_RESIDENT, {"auto": 0, "never": 1, "force": 2}[args.resident])
    if args.wait_timeout_ns:
        c.set_option(skip.SKIP_OPT_WAIT_TIMEOUT_NS, args.wait_timeout_ns)
    reg_d = regions.to(dev)
    off_d = offsets.to(dev)
    out_ids = torch.empty(Q, spec.K, dtype=torch.int64, device=dev)
    out_sc = torch.empty(Q, spec.K, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    ix = None
    if args.ivfpq:
        cent = synth.make_ivf_centroids(spec).to(dev)
        codebook = (synth.train_pq_codebook(spec, args.pq_m, device=dev) if args.pq_train
                    else synth.make_pq_codebook(spec, args.pq_m)).to(dev)
        torch.cuda.synchronize()
        tb = time.perf_counter()
        ix = skip.skip_ivfpq_build(c, cent, codebook)
        build_s = time.perf_counter() - tb
        if args.ivf_refine:
            ix.set_option(skip.SKIP_OPT_IVF_REFINE, args.ivf_refine)

        def step():
            skip.skip_ivfpq_search(ix, reg_d, off_d, args.nprobe, spec.k_region, spec.K, out_ids, out_sc, stream)
    elif args.skv:
        qbar, vbar = synth.make_skv_queries(regions, offsets)
        w1, b1, w2, b2 = synth.make_skv_mlp(spec.d)
        qbar, vbar, w1, b1, w2 = (x.to(dev).contiguous() for x in (qbar, vbar, w1, b1, w2))

        def step():
            return skip.skip_retrieve_skv(c, reg_d, off_d, spec.k_region, spec.K, qbar, vbar, w1, b1, w2, b2,
                                          stream=stream)
    else:
        def step():
            skip.skip_retrieve(c, reg_d, off_d, spec.k_region, spec.K, out_ids, out_sc, stream)

    for _ in range(args.warmup):
        step()
    st = skip.skip_sync_status(c)
    if st != skip.SKIP_OK:
        raise SystemExit("warm-up kernel status: %s" % skip.skip_status_string(st))
    plan = skip.skip_last_plan(c)

    # ---- timed region (device-resident inputs).  Two passes of K steps:
    # the first, with no events between the library's launches, gives the
    # step time (`value`, `ms_per_step`); the second records CUDA events
    # around every launch on the launching stream, for the per-kernel
    # durations (roofline).  Events between launches cost the small
    # workloads several microseconds a step (they break the programmatic
    # overlap of consecutive launches), so they stay out of the first pass.
    timed = ix if ix is not None else c

    def run_timed(with_events):
        timed.set_option(skip.SKIP_OPT_TIMING, 1 if with_events else 0)
        (skip.skip_ivfpq_timing_report(ix) if ix is not None else skip.skip_timing_report(c))
        barrier(world)
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
        barrier(world)
        rep = (skip.skip_ivfpq_timing_report(ix) if ix is not None else skip.skip_timing_report(c))
        timed.set_option(skip.SKIP_OPT_TIMING, 0)
        st = skip.skip_ivfpq_sync_status(ix) if ix is not None else skip.skip_sync_status(c)
        if st != skip.SKIP_OK:
            raise SystemExit("timed kernel status: %s" % skip.skip_status_string(st))
        return e0.elapsed_time(e1), rep

    sampler = ClockSampler(torch.cuda.current_device())
    sampler.start()
    time.sleep(0.3)
    ms_local, _ = run_timed(False)
    clocks = sampler.stop()
    ms_ev_local, kernels = run_timed(True)
    ms = max_over_ranks(ms_local, world)
    ms_ev = max_over_ranks(ms_ev_local, world)
    gate_delta_ms = None
    if args.skv:
        # the gate's cost in the step with its launches overlapped: the same
        # batch with and without the gate, in alternating blocks of steps (so
        # that clock drift under the power cap falls on both alike)
        def plain():
            skip.skip_retrieve(c, reg_d, off_d, spec.k_region, spec.K, out_ids, out_sc, stream)
        for _ in range(args.warmup):
            plain()
        torch.cuda.synchronize()
        # twelve pairs of blocks, the order within a pair alternating; the
        # median of the pairs' differences (a 1 ms step under the power cap
        # wanders by a few us between blocks)
        per = max(1, args.steps // 5)
        diffs = []
        for i in range(12):
            t = {}
            for fn_is_gate in ([False, True] if i % 2 == 0 else [True, False]):
                fn = step if fn_is_gate else plain
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                for _ in range(per):
                    fn()
                e1.record(stream)
                torch.cuda.synchronize()
                t[fn_is_gate] = e0.elapsed_time(e1) / per
            diffs.append(t[True] - t[False])
        gate_delta_ms = max_over_ranks(float(np.median(diffs)), world)

    # ---- end to end through the host-buffer entry point
    reg_h = regions.pin_memory()
    off_h = offsets.pin_memory()
    ids_h = torch.empty(Q, spec.K, dtype=torch.int64).pin_memory()
    sc_h = torch.empty(Q, spec.K, dtype=torch.float32).pin_memory()
    cnt_h = torch.empty(Q, dtype=torch.int32).pin_memory()

    def e2e_step():
        if args.ivfpq:
            reg_d.copy_(reg_h, non_blocking=True)
            off_d.copy_(off_h, non_blocking=True)
            step()
            ids_h.copy_(out_ids, non_blocking=True)
            sc_h.copy_(out_sc, non_blocking=True)
            stream.synchronize()
        elif args.skv:
            # host regions in, gated lists out, through the device entry point
            reg_d.copy_(reg_h, non_blocking=True)
            off_d.copy_(off_h, non_blocking=True)
            g_ids, g_nu, g_cnt = step()
            ids_h.copy_(g_ids, non_blocking=True)
            sc_h.copy_(g_nu, non_blocking=True)
            cnt_h.copy_(g_cnt, non_blocking=True)
            stream.synchronize()
        else:
            skip.skip_retrieve_host(c, reg_h, off_h, spec.k_region, spec.K, ids_h, sc_h, stream)

    for _ in range(3):
        e2e_step()
    barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        e2e_step()
    torch.cuda.synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, world)
    h2d = R * spec.d * 2 + (Q + 1) * 4
    d2h = Q * spec.K * (8 + 4) + (Q * 4 if args.skv else 0)

    # ---- derived figures
    total_q = Q * world * args.steps
    secs = ms / 1e3
    elem = 2 if spec.dtype == "bf16" else 1
    corpus_bytes = spec.N * (spec.d * elem + (4 if spec.dtype == "e4m3" else 0))
    flops = 2.0 * R * spec.N * spec.d
    peaks = load_peaks()
    kname = next((k for k in SCORE_KERNELS if k in kernels), None)
    kinfo = kernels.get(kname, {"launches": 0, "ms": float("nan")})
    k_ms = kinfo["ms"] / max(1, kinfo["launches"])
    t_hbm = corpus_bytes / (peaks["hbm_gbs"] * 1e9)
    t_tc = flops / (peaks["bf16_tflops"] * 1e12)
    if t_tc >= t_hbm:
        achieved = flops / (k_ms / 1e3) / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                "frac": achieved / peaks["bf16_tflops"]}
        if peaks.get("bf16_tflops_sustained"):
            roof["frac_of_sustained"] = achieved / peaks["bf16_tflops_sustained"]
    else:
        achieved = corpus_bytes / (k_ms / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / peaks["hbm_gbs"]}
    traffic = profiled_traffic(kname, spec.name) if kname else None
    roof.update({"traffic": traffic, "kernel": kname, "kernel_ms": k_ms, "peak_source": peaks["source"] +
                 " (MEASURED_PEAKS.json burst)" if peaks["source"] == "measured" else "fallback",
                 "algorithmic_flops_per_launch": flops, "algorithmic_bytes_per_launch": corpus_bytes,
                 "step_roofline_frac": max(t_hbm, t_tc) / (secs / args.steps)})
    if kname and kname + "_bound" in kernels:
        # the bounding pass (every 48th corpus tile first) is extra work of the
        # step, outside the algorithmic count: reported, and in ms_per_step
        kb = kernels[kname + "_bound"]
        roof["bound_pass_ms"] = kb["ms"] / max(1, kb["launches"])
        roof["frac_with_bound_pass"] = roof["frac"] * k_ms / (k_ms + roof["bound_pass_ms"])
        roof["kernel_note"] = ("frac: full pass only; each call first runs a bounding pass over every 48th "
                               "corpus tile (bound_pass_ms, counted in ms_per_step); frac_with_bound_pass: the "
                               "algorithmic work over both passes' time")
    line = {
        "metric": METRIC, "value": total_q / secs, "unit": "queries/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
        "ms_per_step_with_kernel_events": ms_ev / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic", "config": workload_config(spec, R, world),
        "corpus_gbs": corpus_bytes * world * args.steps / secs / 1e9,
        "region_rows_per_s": R * world * args.steps / secs,
        "tflops": flops * world * args.steps / secs / 1e12,
        "roofline": roof,
        "clocks": clocks,
        "e2e": {"value": total_q / e2e_s, "unit": "queries/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h,
                "entry_point": ("skip_ivfpq_search with pinned host copies in and out" if args.ivfpq else
                                "skip_retrieve_skv with pinned host copies in and out" if args.skv
                                else "skip_retrieve_host (pinned host buffers)")},
        # kernels counted in the events pass; without events the SKV gate's
        # bias GEMM runs on a second stream followed by its one-thread ready
        # flag kernel, one more launch a step
        "gpu_launches": int(sum(v["launches"] for v in kernels.values())) + (args.steps if args.skv else 0),
        "kernels": kernels,
        "plan": plan,
        "dedup_rate": None if args.ivfpq else dedup_rate(skip, c, reg_d, offsets, spec.k_region),
    }
    if args.ivfpq:
        line.update(ivfpq_report(args, spec, skip, c, ix, cent, reg_d, off_d, kernels, build_s, peaks, ms))
        line["config"]["variant"] = "IVF-PQ: %d centroids, PQ%d, nprobe %d%s" % (
            cent.shape[0], args.pq_m, args.nprobe,
            ", exact re-rank of the best %d x k_region" % args.ivf_refine if args.ivf_refine else "")
        ix.free()
    if args.skv:
        line["config"]["skv_gate"] = {"hidden": 512, "tau_nu": 0.5, "rho_r": 0.6}
        H = 512
        P = Q * spec.K
        skv_flops = 2.0 * P * 3 * spec.d * H + 2.0 * Q * 2 * spec.d * H
        skv_ms = sum(kernels[k]["ms"] / max(1, kernels[k]["launches"]) for k in kernels if k.startswith("skv_"))
        mlp = kernels.get("skv_mlp", {"ms": float("nan"), "launches": 1})
        mlp_ms = mlp["ms"] / max(1, mlp["launches"])
        line["skv"] = {"gate_ms_per_step": skv_ms, "mlp_kernel_ms": mlp_ms,
                       "gate_step_delta_ms": gate_delta_ms,
                       "mlp_algorithmic_flops": 2.0 * P * 3 * spec.d * H,
                       "mlp_tflops": 2.0 * P * 3 * spec.d * H / (mlp_ms / 1e3) / 1e12,
                       "gate_share_of_step": skv_ms / (ms / args.steps), "algorithmic_flops": skv_flops}
    if keep_host:
        line["cpu_baseline"] = cpu_baseline(spec, corpus_np, scale_np, regions, offsets, args.cpu_questions)
    c.free()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
