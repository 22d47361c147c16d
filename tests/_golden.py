"""Reader for the text fixtures under tests/golden/."""
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def read_fixture(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        lines = [ln.strip() for ln in f if ln.strip() and not ln.lstrip().startswith("#")]
    i = 0
    while i < len(lines):
        parts = lines[i].split()
        key = parts[0]
        if len(parts) == 2 and key in ("corpus", "regions", "region_ids", "region_scores",
                                       "merged_ids", "merged_scores", "skv_corpus", "w1", "qbar",
                                       "vbar", "ids", "nu_all", "out_ids", "out_nu", "centroids",
                                       "codebook", "ivf_corpus", "queries", "codes", "p1k2_ids",
                                       "p1k2_scores", "p1k4_ids", "p1k4_scores", "p2k3_ids",
                                       "p2k3_scores", "qvs_tokens", "wv", "hv", "hk", "qh", "kh", "vh",
                                       "out1", "out2"):
            n = int(parts[1])
            rows = [[float(v) for v in lines[i + 1 + t].split()] for t in range(n)]
            out[key] = np.array(rows, dtype=np.float64)
            i += 1 + n
        else:
            vals = [float(v) for v in parts[1:]]
            out[key] = vals[0] if len(vals) == 1 else np.array(vals)
            i += 1
    return out
