"""The fixed-radius search's traversal, walked on the CPU: hits sorted by their cell on a grid over
the first K embedding coordinates (cells 0.1 % wider than half the radius), each hit visiting the
rows of cells at or after its own in key order (runs of five cells along the last gridded axis),
must find every pair within the radius exactly once.  Checked against a brute-force scan with the
same fp32 distance rule, on random unit vectors and on pairs placed at the radius across cell
boundaries.  (This is the index logic of the search, not its kernel: the GPU result is compared
with the oracle in tests/test_gpu_graph.py.)"""
import itertools

import numpy as np
import pytest

from oracle import gnn_oracle as O

REACH = 2


def grid_cells(radius, K):
    cells = np.float32(1.998 * REACH) / np.float32(radius)
    cap = 64 if K == 4 else 128
    return cap if cells >= cap else (1 if cells < 1 else int(cells))


def traverse(emb, radius):
    emb = np.asarray(emb, np.float32)
    n, dim = emb.shape
    K = 4 if dim >= 4 else 3
    g = grid_cells(radius, K)
    c = np.zeros((n, K), np.int64)
    for k in range(min(K, dim)):
        c[:, k] = np.clip(np.floor((emb[:, k] + np.float32(1)) * np.float32(0.5) * np.float32(g)), 0, g - 1)
    key = np.zeros(n, np.int64)
    for k in range(K):
        key = key * g + c[:, k]
    ids = np.argsort(key, kind="stable")
    ks = key[ids]
    start = np.searchsorted(ks, np.arange(g ** K + 1))
    es = emb[ids]
    r2 = np.float32(np.float32(radius) * np.float32(radius))
    offsets = [o for o in itertools.product(range(-REACH, REACH + 1), repeat=K - 1) if o >= (0,) * (K - 1)]
    found = []
    for t in range(n):
        cell = c[ids[t]]
        lo, hi = max(cell[-1] - REACH, 0), min(cell[-1] + REACH, g - 1)
        for off in offsets:
            row_c = cell[:-1] + np.asarray(off, np.int64)
            if np.any(row_c < 0) or np.any(row_c >= g):
                continue
            row = 0
            for v in row_c:
                row = row * g + int(v)
            row *= g
            p0 = t + 1 if all(o == 0 for o in off) else start[row + lo]
            p1 = start[row + hi + 1]
            if p1 <= p0:
                continue
            d = O.sq_dist_f32(np.broadcast_to(es[t], (p1 - p0, dim)), es[p0:p1])
            for q in np.flatnonzero(d < r2) + p0:
                found.append(tuple(sorted((int(ids[t]), int(ids[q])))))
    return found


def brute(emb, radius):
    emb = np.asarray(emb, np.float32)
    ii, jj = np.triu_indices(emb.shape[0], 1)
    r2 = np.float32(np.float32(radius) * np.float32(radius))
    keep = O.sq_dist_f32(emb[ii], emb[jj]) < r2
    return sorted(zip(ii[keep].tolist(), jj[keep].tolist()))


@pytest.mark.parametrize("dim,radius", [(3, 0.3), (8, 0.45), (5, 0.35), (2, 0.1), (8, 2.5)])
def test_traversal_finds_each_pair_once(dim, radius):
    rng = np.random.default_rng(dim)
    e = rng.standard_normal((600, dim))
    e /= np.linalg.norm(e, axis=1, keepdims=True)
    got = traverse(e, radius)
    assert len(got) == len(set(got))                              # once
    assert sorted(got) == brute(e, radius)                        # every pair


def test_pairs_at_the_radius_across_cell_boundaries():
    """Pairs just inside and just outside the radius, straddling cell edges on every gridded axis."""
    rng = np.random.default_rng(0)
    radius = np.float32(0.2)
    g = grid_cells(radius, 4)
    w = 2.0 / g
    pts = []
    for _ in range(150):
        base = -1 + w * rng.integers(1, g - 1, size=8)             # on a cell boundary
        base[4:] = rng.uniform(-0.5, 0.5, 4)
        d = rng.standard_normal(8)
        d /= np.linalg.norm(d)
        for scale in (0.999, 1.0, 1.001):
            pts.append(base - 0.5 * scale * float(radius) * d)
            pts.append(base + 0.5 * scale * float(radius) * d)
    e = np.asarray(pts, np.float32)
    got = traverse(e, radius)
    assert len(got) == len(set(got)) and sorted(got) == brute(e, radius)
