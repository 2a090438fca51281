"""Embedding and graph building on the GPU (gnn_embed_load / gnn_embed / gnn_build_graph through the
C ABI), and the whole pipeline of the paper's Section 2.1 on one event: embedding -> fixed-radius
graph -> filtering -> interaction network -> track labels.  Where a float decides an integer (an edge
inside the radius, a score above a threshold) both sides decide on the GPU's values."""
import numpy as np
import pytest

from oracle import gnn_oracle as O
from paper_2402_09633_gb300 import synthetic as S
from tests.gpu_util import check_parity

pytestmark = pytest.mark.gpu
DIM = 8


def _net(cfg, dim=DIM):
    from paper_2402_09633_gb300 import InteractionNetwork
    W = S.init_weights(cfg, 0)
    ew = S.init_embed_weights(cfg, dim, 2)
    net = InteractionNetwork(cfg, S.pack_blob(cfg, W))
    net.load_embedding(S.pack_embed_blob(cfg, ew))
    return net, W, ew


def _radius_for(emb, k=4):
    """A radius giving about k neighbours per hit (median distance to the k-th neighbour)."""
    kd = pytest.importorskip("scipy.spatial")
    d, _ = kd.cKDTree(emb.astype(np.float64)).query(emb.astype(np.float64), k + 1)
    return float(np.median(d[:, k]))


def _oracle_graph(emb, r_col, radius):
    kd = pytest.importorskip("scipy.spatial")
    cand = np.array(sorted(kd.cKDTree(emb.astype(np.float64)).query_pairs(radius * 1.001)), np.int64).reshape(-1, 2)
    return O.radius_graph(emb, r_col, radius, cand)


def _sorted_edges(ei):
    e = np.asarray(ei).T.astype(np.int64)
    return e[np.lexsort((e[:, 1], e[:, 0]))]


@pytest.mark.parametrize("H,L", [(128, 3), (64, 2)])
def test_embedding_matches_oracle(H, L):
    import torch
    cfg = S.ModelConfig(12, 2, H, 2, L)
    net, _, ew = _net(cfg)
    x, _ = S.generate_event(S.EventSpec(30000, 9, "powerlaw", 0.02, n_edges=100000), 1)
    got = net.embed(torch.from_numpy(x).cuda()).cpu().numpy()
    want = O.embed(ew, x, cfg.ln_eps)
    assert np.abs(got - want).max() < 2e-4
    np.testing.assert_allclose(np.linalg.norm(got, axis=1), 1.0, atol=1e-5)
    assert net.status() == 0
    net.close()


def _event_graph(net, n, seed, k=4):
    import torch
    x, _ = S.generate_event(S.EventSpec(n, 9, "powerlaw", 0.02, n_edges=n * 3), seed)
    xs = torch.from_numpy(x).cuda()
    emb = net.embed(xs)
    e_np = emb.cpu().numpy()
    radius = _radius_for(e_np if n <= 30000 else e_np[:30000], k) * (1.0 if n <= 30000 else 0.7)
    ei, m = net.build_graph(emb, xs, radius, max_edges=40 * n)
    ei2, m2 = net.build_graph(emb, xs, radius, max_edges=40 * n)
    assert m == m2 and ei.cpu().numpy().tobytes() == ei2.cpu().numpy().tobytes()     # deterministic
    return x, e_np, radius, ei.cpu().numpy(), m


@pytest.mark.parametrize("n", [2000, 30000])
def test_radius_graph_matches_oracle(n):
    cfg = S.ModelConfig(12, 2, 128, 2, 3)
    net, _, _ = _net(cfg)
    x, e_np, radius, ei, m = _event_graph(net, n, 2)
    got = _sorted_edges(ei)
    assert got.shape[0] == m and m > n
    np.testing.assert_array_equal(got, _oracle_graph(e_np, x[:, 0], radius))
    net.close()


@pytest.mark.parametrize("dim", [2, 5, 12])
def test_radius_graph_other_embedding_widths(dim):
    """D = 2 (grid over 3 coordinates, two of them real), 5 and 12 (grid over 4; one, two and three
    float4 chunks per sorted embedding): edge sets bit-exact against the oracle."""
    import torch
    cfg = S.ModelConfig(12, 2, 64, 2, 2)
    net, _, ew = _net(cfg, dim=dim)
    x, _ = S.generate_event(S.EventSpec(4000, 9, "powerlaw", 0.02, n_edges=12000), 5)
    xs = torch.from_numpy(x).cuda()
    emb = net.embed(xs)
    e_np = emb.cpu().numpy()
    assert e_np.shape == (4000, dim)
    np.testing.assert_allclose(e_np, O.embed(ew, x, cfg.ln_eps), atol=2e-4)
    radius = _radius_for(e_np, 4)
    ei, m = net.build_graph(emb, xs, radius, max_edges=200 * 4000)
    assert m > 0
    np.testing.assert_array_equal(_sorted_edges(ei.cpu().numpy()), _oracle_graph(e_np, x[:, 0], radius))
    net.close()


def test_partner_chains_and_search_again_agree():
    """The counting pass keeps each hit's partners in chains of 15-entry chunks that the writing pass
    copies; a hit whose chain could not grow (pool used up) is searched again.  At a radius giving
    about 40 neighbours per hit (chains of several chunks), the default pool, an empty pool and a
    pool that runs out part-way give byte-identical edge lists, equal to the oracle's edge set."""
    import ctypes
    import torch
    cfg = S.ModelConfig(12, 2, 64, 2, 2)
    net, _, _ = _net(cfg)
    n = 8000
    x, _ = S.generate_event(S.EventSpec(n, 9, "powerlaw", 0.02, n_edges=3 * n), 4)
    xs = torch.from_numpy(x).cuda()
    emb = net.embed(xs)
    e_np = emb.cpu().numpy()
    radius = _radius_for(e_np, 40)
    net.lib.gnn_debug_graph_pool.argtypes = [ctypes.c_void_p, ctypes.c_int64]
    net.lib.gnn_debug_graph_pool.restype = ctypes.c_int
    outs = []
    for pool in (-1, 0, 100):
        assert net.lib.gnn_debug_graph_pool(net.handle, pool) == 0
        ei, m = net.build_graph(emb, xs, radius, max_edges=100 * n)
        assert net.status() == 0
        outs.append(ei.cpu().numpy().tobytes())
    assert outs[0] == outs[1] == outs[2]
    got = _sorted_edges(np.frombuffer(outs[0], np.int32).reshape(2, -1))
    assert got.shape[0] > 15 * n                       # more than one chunk per hit on average
    np.testing.assert_array_equal(got, _oracle_graph(e_np, x[:, 0], radius))
    assert net.lib.gnn_debug_graph_pool(None, 0) == -1
    net.close()


def test_radius_graph_full_event_sampled():
    """300k hits: the edges of 400 sampled hits against a brute-force search over every hit, and
    the properties every edge list must have (no self-loops, no duplicates, oriented by r)."""
    cfg = S.ModelConfig(12, 2, 128, 2, 3)
    net, _, _ = _net(cfg)
    n = 300000
    x, e_np, radius, ei, m = _event_graph(net, n, 3)
    assert m > n // 4
    src, dst = ei[0].astype(np.int64), ei[1].astype(np.int64)
    assert np.all(src != dst) and np.unique(np.minimum(src, dst) * n + np.maximum(src, dst)).size == m
    r = x[:, 0]
    assert np.all((r[src] < r[dst]) | ((r[src] == r[dst]) & (src < dst)))
    r2 = np.float32(np.float32(radius) * np.float32(radius))
    for i in np.random.default_rng(0).choice(n, 400, replace=False):
        d = O.sq_dist_f32(np.broadcast_to(e_np[i], e_np.shape), e_np)
        want = np.flatnonzero(d < r2)
        want = want[want != i]
        got = np.sort(np.concatenate([dst[src == i], src[dst == i]]))
        np.testing.assert_array_equal(got, want)
    net.close()


def test_graph_capacity_and_degenerate_inputs():
    import torch
    from paper_2402_09633_gb300 import GnnError
    cfg = S.ModelConfig(3, 2, 64, 1, 2)
    net, _, _ = _net(cfg, dim=3)
    x, _ = S.random_graph(3000, 0, 3, 4)
    xs = torch.from_numpy(x).cuda()
    emb = net.embed(xs)
    ei, k = net.build_graph(emb, xs, 0.05, max_edges=10 ** 6)
    assert k > 3000
    with pytest.raises(GnnError) as ex:                        # not enough room: nothing written, code CAPACITY
        net.build_graph(emb, xs, 0.05, max_edges=k - 1)
    assert ex.value.code == -7 and ex.value.n_edges == k
    assert net.status() == 0
    ei2, k2 = net.build_graph(emb, xs, 0.05, max_edges=k)      # exactly enough
    assert k2 == k and ei2.cpu().numpy().tobytes() == ei.cpu().numpy().tobytes()
    _, k0 = net.build_graph(emb, xs, 1e-6, max_edges=10)       # tiny radius: no pairs
    assert k0 == 0
    _, kall = net.build_graph(emb[:50].contiguous(), xs[:50].contiguous(), 2.5, max_edges=2000)
    assert kall == 50 * 49 // 2                                 # radius beyond the sphere's diameter
    net.close()


def test_whole_pipeline_on_one_event():
    """Embedding -> graph -> filtering -> interaction network -> track labels, each stage checked
    against the oracle fed with the previous GPU stage's output."""
    import torch
    cfg = S.ModelConfig(12, 2, 128, 3, 3)
    net, W, ew = _net(cfg)
    fw = S.init_filter_weights(cfg, 5)
    net.load_filter(S.pack_filter_blob(cfg, fw))
    x, _ = S.generate_event(S.EventSpec(30000, 9, "powerlaw", 0.02, n_edges=100000), 7)
    xs = torch.from_numpy(x).cuda()
    emb = net.embed(xs)
    e_np = emb.cpu().numpy()
    np.testing.assert_allclose(e_np, O.embed(ew, x, cfg.ln_eps), atol=2e-4)
    radius = _radius_for(e_np, 3)
    cand, k = net.build_graph(emb, xs, radius, max_edges=10 ** 6)
    np.testing.assert_array_equal(_sorted_edges(cand.cpu().numpy()), _oracle_graph(e_np, x[:, 0], radius))
    cand = cand.contiguous()
    fsc, kept, ids = net.filter_edges(xs, cand, float(np.median(O.filter_scores(fw, x, cand.cpu().numpy()))))
    kept = kept.contiguous()
    assert 0 < kept.shape[1] < k
    scores = net.infer(xs, kept)
    labels = net.track_labels(scores, kept, x.shape[0], 0.5)
    assert net.status() == 0
    k_np, s_np = kept.cpu().numpy(), scores.cpu().numpy()
    check_parity(s_np, W, x, k_np, cfg.n_iters)
    np.testing.assert_array_equal(labels.cpu().numpy(), O.track_labels(s_np, k_np, x.shape[0], 0.5))
    net.close()
