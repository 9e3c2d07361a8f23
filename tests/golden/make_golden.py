"""Writes the tiny-workload regression fixtures from the fp64 oracle.

Calls only oracle/ and the seeded input generators (no CUDA code):
  tiny_projected.txt  [8, 256] unnormalised projected gradients
  tiny_topk.txt       top-4 store rows (index, cosine score) for 8 queries
"""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

from oracle import bergson_oracle as orc  # noqa: E402
from paper_2606_11660_gb300 import workloads as wl  # noqa: E402

TOPK = 4
QUERY_SEED = 3


def tiny_layers():
    """The tiny workload: seeds as the tests' make_layers(..., rc=True) draws them."""
    cfg = wl.TINY
    spec = cfg.modules[0]
    A, G = wl.layer_inputs(spec, cfg.B, cfg.T, seed=0)
    r, c = wl.second_moments(spec.d_out, spec.d_in, seed=500)
    s_in, s_out = orc.module_seeds(0, 0)
    layer = orc.Layer(A.float().numpy(), G.float().numpy(), cfg.k, cfg.k, s_in, s_out,
                      r.numpy().astype(np.float64), c.numpy().astype(np.float64), 0)
    return cfg, [layer]


def compute():
    cfg, layers = tiny_layers()
    proj = orc.project_grads(layers, None, cfg.k * cfg.k)
    store, _ = orc.build_store(proj)
    queries = wl.gaussian_rows(cfg.B, cfg.k * cfg.k, seed=QUERY_SEED).numpy().astype(np.float64)
    scores, idx = orc.score_topk(store, queries, TOPK)
    return proj, scores, idx


def main():
    proj, scores, idx = compute()
    with open(os.path.join(HERE, "tiny_projected.txt"), "w") as f:
        f.write("# tiny workload: oracle projected gradients [8, 256] (fp64, row per example)\n")
        for row in proj:
            f.write(" ".join(f"{v:.17g}" for v in row) + "\n")
    with open(os.path.join(HERE, "tiny_topk.txt"), "w") as f:
        f.write(f"# tiny workload store vs 8 N(0, I) queries (seed {QUERY_SEED}): "
                f"top-{TOPK} as index:score per query\n")
        for q in range(idx.shape[0]):
            f.write(" ".join(f"{int(i)}:{s:.17g}" for i, s in zip(idx[q], scores[q])) + "\n")


if __name__ == "__main__":
    main()
