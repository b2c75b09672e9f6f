"""Writes the stored oracle outputs under tests/golden/ (calls only the oracle
and the seeded input generator).

    python tests/golden/make_golden.py

tiny_fp32_oracle.txt: for the 1-request, 1-layer, d=64 workload (seed 20261):
the LOCAL_GLOBAL and FULL logits and probabilities of all 16 candidates, the
pooled anchor g, the first cached K row of layer 0, and the scores after the
4-row incremental append.  A later change of these values must come with the
passage of the paper (or its reading) that justifies the oracle change.
"""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

from oracle import txs_oracle as O  # noqa: E402
from paper_2607_28940_gb300 import workload as W  # noqa: E402


def tiny_values():
    wl = W.WORKLOADS["tiny_fp32"]
    model = O.Model.from_arrays(W.weights(wl), wl)
    b = W.batch(wl)
    caches = O.build_caches(model, b.beh, b.beh_off)
    out = {}
    for name, mode in (("local_global", O.LOCAL_GLOBAL), ("full", O.FULL)):
        lg, pr = O.score_batch(model, caches, b.ctx, b.cand, b.cand_off, mode)
        out[f"{name}.logits"] = lg
        out[f"{name}.probs"] = pr
    out["anchor_g"] = caches[0].pool.g[None]
    out["K0_row0"] = caches[0].K[0][:1]
    app = O.append_caches(model, caches, b.app, b.app_off)
    lg, pr = O.score_batch(model, app, b.ctx, b.cand, b.cand_off, O.LOCAL_GLOBAL)
    out["appended.local_global.logits"] = lg
    return out


def write(path, values):
    with open(path, "w") as f:
        f.write("# oracle outputs, tiny_fp32 workload; written by tests/golden/make_golden.py\n")
        for k, v in values.items():
            v = np.atleast_2d(v)
            f.write(f"{k} {v.shape[0]} {v.shape[1]}\n")
            for row in v:
                f.write(" ".join(f"{x:.17g}" for x in row) + "\n")


def read(path):
    vals = {}
    with open(path) as f:
        lines = [l for l in f.read().splitlines() if l and not l.startswith("#")]
    i = 0
    while i < len(lines):
        name, n, m = lines[i].split()
        n, m = int(n), int(m)
        vals[name] = np.array([[float(x) for x in lines[i + 1 + j].split()] for j in range(n)])
        i += 1 + n
    return vals


if __name__ == "__main__":
    write(os.path.join(HERE, "tiny_fp32_oracle.txt"), tiny_values())
