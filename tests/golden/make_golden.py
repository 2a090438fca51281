"""Writes tests/golden/oracle_small_logits.txt by calling only the oracle.

The stored logits pin the oracle against unintended later changes; they are
the oracle's own fp64 output on a fixed seeded graph (120 nodes, 400 edges,
H=16, 2-layer MLPs, T=3), not values printed in the paper (it prints none)."""
import os
import sys

import numpy as np

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))))
from oracle import gnn_oracle as O                       # noqa: E402
from paper_2402_09633_gb300 import synthetic as S        # noqa: E402


def golden_case():
    cfg = S.ModelConfig(3, 2, 16, 3, 2)
    W = S.init_weights(cfg, seed=11)
    x, ei = S.random_graph(120, 400, 3, seed=12)
    return W, x, ei, cfg.n_iters


if __name__ == "__main__":
    W, x, ei, T = golden_case()
    _, logits = O.forward(W, x, ei, T, return_logits=True)
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_small_logits.txt")
    np.savetxt(out, logits, fmt="%.17g")
    print("wrote", out, logits.shape)
