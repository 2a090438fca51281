"""Filtering step on the GPU (gnn_filter_load / gnn_filter_edges through the C ABI): the filter
MLP's scores against the oracle (fp32 model: logits within 2e-3), the kept edge list bit-exact
against applyFiltering of the same (GPU) scores, and the chain filter -> GNN -> track labels."""
import numpy as np
import pytest

from oracle import gnn_oracle as O
from paper_2402_09633_gb300 import synthetic as S
from tests.gpu_util import LOGIT_TOL_FP32, check_parity, logits_from_scores

pytestmark = pytest.mark.gpu


def _net(cfg, seed=0, fseed=1):
    from paper_2402_09633_gb300 import InteractionNetwork
    W = S.init_weights(cfg, seed)
    fw = S.init_filter_weights(cfg, fseed)
    net = InteractionNetwork(cfg, S.pack_blob(cfg, W))
    net.load_filter(S.pack_filter_blob(cfg, fw))
    return net, W, fw


def _filter(net, x, ei, thr):
    import torch
    sc, kept, ids = net.filter_edges(torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda(), thr)
    return sc.cpu().numpy(), kept.cpu().numpy(), ids.cpu().numpy()


def _check_kept(sc, kept, ids, ei, thr):
    want_kept, want_ids = O.apply_filtering(sc, ei, thr)
    np.testing.assert_array_equal(ids, want_ids)
    np.testing.assert_array_equal(kept, want_kept)


@pytest.mark.parametrize("H,L", [(128, 3), (64, 2)])
def test_filter_scores_and_kept_edges(H, L):
    cfg = S.ModelConfig(12, 2, H, 2, L)
    net, _, fw = _net(cfg)
    x, ei = S.generate_event(S.EventSpec(30000, 9, "powerlaw", 0.02, n_edges=100000), 4)
    ref, want = O.filter_scores(fw, x, ei, cfg.ln_eps, return_logits=True)
    for thr in np.quantile(ref, [0.25, 0.5, 0.75]).tolist():   # a random-init filter: its own quartiles
        sc, kept, ids = _filter(net, x, ei, thr)
        err = np.abs(logits_from_scores(sc) - want)
        assert err.max() <= LOGIT_TOL_FP32, f"max filter logit error {err.max():.3e}"
        _check_kept(sc, kept, ids, ei, thr)
        assert 0 < ids.size < ei.shape[1]
    assert net.status() == 0
    net.close()


def test_filter_bf16_model():
    cfg = S.ModelConfig(12, 2, 128, 2, 3, S.PRECISION_BF16)
    net, _, fw = _net(cfg)
    x, ei = S.generate_event(S.EventSpec(3000, 9, "powerlaw", 0.02, n_edges=10007), 5)
    ref, z64 = O.filter_scores(fw, x, ei, cfg.ln_eps, bf16=True, return_logits=True)
    thr = float(np.median(ref))
    sc, kept, ids = _filter(net, x, ei, thr)
    err = np.abs(logits_from_scores(sc) - z64)
    assert err.max() <= 1e-2, f"max filter logit error {err.max():.3e}"
    _check_kept(sc, kept, ids, ei, thr)
    net.close()


def test_filter_edge_cases():
    import torch
    cfg = S.ModelConfig(3, 2, 64, 1, 2)
    net, _, fw = _net(cfg)
    x, ei = S.random_graph(200, 1000, 3, 6)
    sc, kept, ids = _filter(net, x, ei, -1.0)                  # every edge kept
    assert ids.tolist() == list(range(1000)) and np.array_equal(kept, ei)
    sc2, kept, ids = _filter(net, x, ei, 2.0)                  # none kept
    assert ids.size == 0 and kept.shape == (2, 0) and sc2.tobytes() == sc.tobytes()
    sc, kept, ids = _filter(net, x, np.zeros((2, 0), np.int32), 0.5)
    assert sc.size == 0 and ids.size == 0
    bad = ei.copy(); bad[1, 5] = 200; bad[0, 9] = -1           # endpoints out of range
    sc, kept, ids = _filter(net, x, bad, -1.0)
    assert np.isnan(sc[5]) and np.isnan(sc[9]) and 5 not in ids and 9 not in ids and ids.size == 998
    assert net.status() == -5 and net.status() == 0
    net.close()


def test_filter_blob_validation():
    from paper_2402_09633_gb300 import GnnError, InteractionNetwork
    cfg = S.ModelConfig(3, 2, 64, 1, 2)
    net = InteractionNetwork(cfg, S.pack_blob(cfg, S.init_weights(cfg, 0)))
    import torch
    x, ei = S.random_graph(10, 20, 3, 0)
    with pytest.raises(GnnError) as ex:                        # no filter loaded yet
        net.filter_edges(torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda())
    assert ex.value.code == -1
    blob = S.pack_filter_blob(cfg, S.init_filter_weights(cfg, 1))
    for b in (b"XXXX" + blob[4:], blob[:-4],
              S.pack_filter_blob(S.ModelConfig(3, 2, 128, 1, 2), S.init_filter_weights(S.ModelConfig(3, 2, 128, 1, 2))),
              S.pack_filter_blob(S.ModelConfig(4, 2, 64, 1, 2), S.init_filter_weights(S.ModelConfig(4, 2, 64, 1, 2)))):
        with pytest.raises(GnnError) as ex:
            net.load_filter(b)
        assert ex.value.code == -2
    net.load_filter(blob)
    net.close()


def test_filter_then_gnn_then_track_labels():
    """The service chain of the paper's pipeline tail on one event: filtering MLP + applyFiltering,
    interaction network on the kept edges, track labels from its scores."""
    import torch
    cfg = S.ModelConfig(12, 2, 128, 3, 3)
    net, W, fw = _net(cfg, 2, 3)
    x, ei = S.generate_event(S.EventSpec(30000, 9, "powerlaw", 0.02, n_edges=100000), 6)
    xs = torch.from_numpy(x).cuda()
    thr = float(np.median(O.filter_scores(fw, x, ei, cfg.ln_eps)))
    fsc, kept, ids = net.filter_edges(xs, torch.from_numpy(ei).cuda(), thr)
    kept = kept.contiguous()
    scores = net.infer(xs, kept)
    labels = net.track_labels(scores, kept, x.shape[0], 0.5)
    assert net.status() == 0
    k_np, s_np = kept.cpu().numpy(), scores.cpu().numpy()
    _check_kept(fsc.cpu().numpy(), k_np, ids.cpu().numpy(), ei, thr)
    assert 0.3 * ei.shape[1] < k_np.shape[1] < 0.7 * ei.shape[1]
    check_parity(s_np, W, x, k_np, cfg.n_iters)
    np.testing.assert_array_equal(labels.cpu().numpy(), O.track_labels(s_np, k_np, x.shape[0], 0.5))
    net.close()
