"""Track candidates on the GPU (gnn_track_labels through the C ABI): bit-exact labels against the
oracle's connected components of the same thresholded edges.  Where a score decides whether an edge
is kept, both sides decide on the same (GPU) score."""
import numpy as np
import pytest

from oracle import gnn_oracle as O
from paper_2402_09633_gb300 import synthetic as S

pytestmark = pytest.mark.gpu


def _net():
    from paper_2402_09633_gb300 import InteractionNetwork
    cfg = S.ModelConfig(3, 2, 64, 1, 2)
    return InteractionNetwork(cfg, S.pack_blob(cfg, S.init_weights(cfg, 0)))


def _gpu_labels(net, scores, ei, n, thr):
    import torch
    lab = net.track_labels(torch.from_numpy(np.ascontiguousarray(scores, np.float32)).cuda(),
                           torch.from_numpy(np.ascontiguousarray(ei, np.int32)).cuda(), n, thr)
    assert net.status() == 0
    return lab.cpu().numpy()


@pytest.mark.parametrize("n,m,seed", [(1, 0, 0), (10, 40, 1), (1000, 700, 2), (1000, 3000, 3),
                                      (200000, 150000, 4), (200000, 1000000, 5)])
def test_labels_match_oracle_on_random_graphs(n, m, seed):
    rng = np.random.default_rng(seed)
    ei = rng.integers(0, n, size=(2, m)).astype(np.int32)
    sc = rng.random(m).astype(np.float32)
    net = _net()
    for thr in (0.2, 0.5, 0.95):
        np.testing.assert_array_equal(_gpu_labels(net, sc, ei, n, thr), O.track_labels(sc, ei, n, thr))
    net.close()


def test_long_chains_and_stars():
    """Worst cases for union-find: one long path in shuffled order, and a star."""
    rng = np.random.default_rng(7)
    n = 300000
    order = rng.permutation(n)
    ei = np.stack([order[:-1], order[1:]]).astype(np.int32)[:, rng.permutation(n - 1)]
    star = np.stack([np.full(n - 1, n // 2), np.delete(np.arange(n), n // 2)]).astype(np.int32)
    net = _net()
    for e in (ei, star):
        sc = np.ones(e.shape[1], np.float32)
        lab = _gpu_labels(net, sc, e, n, 0.5)
        assert (lab == 0).all()
    net.close()


def test_special_edges_are_skipped():
    ei = np.array([[0, 1, 3, 4, 2, -1], [1, 2, 3, 9, 7, 0]], np.int32)   # self-loop, out of range
    sc = np.array([0.9, 0.9, 0.9, 0.9, np.nan, 0.9], np.float32)
    net = _net()
    assert _gpu_labels(net, sc, ei, 6, 0.5).tolist() == [0, 0, 0, 3, 4, 5]
    assert _gpu_labels(net, np.zeros(0, np.float32), np.zeros((2, 0), np.int32), 4, 0.5).tolist() == [0, 1, 2, 3]
    net.close()


def test_full_event_scores_to_track_labels():
    """The whole service path on the benchmark event: scores from gnn_infer, then labels."""
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    w = S.WORKLOADS["full"]
    x, ei = S.generate_event(w.event, 0)
    net = InteractionNetwork(w.model, S.pack_blob(w.model, S.init_weights(w.model, w.weight_seed)))
    xs, es = torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda()
    scores = net.infer(xs, es)
    lab1 = net.track_labels(scores, es, x.shape[0], 0.5).cpu().numpy()
    lab2 = net.track_labels(scores, es, x.shape[0], 0.5).cpu().numpy()
    assert net.status() == 0
    s = scores.cpu().numpy()
    np.testing.assert_array_equal(lab1, O.track_labels(s, ei, x.shape[0], 0.5))
    assert lab1.tobytes() == lab2.tobytes()
    n_tracks = np.unique(lab1).size
    print(f"full event: {int((s > 0.5).sum())} kept edges, {n_tracks} components")
    net.close()
