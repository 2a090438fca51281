"""GPU parity: the CUDA path through the C ABI against the fp64 CPU oracle.

Integer outputs (CSR) are compared bit-exactly; scores are compared as logits
with the max-abs tolerance of the fp32 path (2e-3) plus decision agreement at
the 0.5 threshold wherever the oracle logit is more than 1e-2 from it."""
import numpy as np
import pytest

from oracle import gnn_oracle as O
from paper_2402_09633_gb300 import synthetic as S
from tests.gpu_util import check_parity, run_gpu, untile

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("n,e,seed", [(1, 1, 0), (5, 3, 1), (300, 4096, 2), (1000, 4097, 3),
                                       (70000, 250001, 4), (3, 20000, 5)])
def test_csr_bit_exact(n, e, seed):
    import torch
    cfg = S.ModelConfig(3, 2, 64, 1, 2)
    W = S.init_weights(cfg, 0)
    x, ei = S.random_graph(n, e, 3, seed)
    _, rc, net = run_gpu(cfg, W, x, ei, return_net=True)
    assert rc == 0
    rowptr, src_sorted, perm = O.csr_by_destination(ei[0], ei[1], n)
    got_rowptr = net.debug_copy(0, (n + 1,), torch.int32).cpu().numpy()
    got_perm = net.debug_copy(1, (e,), torch.int32).cpu().numpy()
    got_src = net.debug_copy(2, (e,), torch.int32).cpu().numpy()
    net.close()
    np.testing.assert_array_equal(got_rowptr, rowptr)
    np.testing.assert_array_equal(got_perm, perm)
    np.testing.assert_array_equal(got_src, src_sorted)


@pytest.mark.parametrize("T", [0, 1, 3])
def test_small_graph_parity_h128(T):
    cfg = S.ModelConfig(3, 2, 128, T, 3)
    W = S.init_weights(cfg, 7)
    x, ei = S.generate_event(S.EventSpec(2000, 0, "fanout", 0.3), 1)   # ragged last tile
    s, rc = run_gpu(cfg, W, x, ei)
    assert rc == 0
    check_parity(s, W, x, ei, T)


def test_node_state_after_iterations():
    """Node states h after T iterations match the oracle's (fp32 tolerance)."""
    import torch
    cfg = S.ModelConfig(12, 2, 128, 2, 3)
    W = S.init_weights(cfg, 3)
    x, ei = S.generate_event(S.EventSpec(3000, 9, "powerlaw", 0.02, n_edges=10007), 2)
    s, rc, net = run_gpu(cfg, W, x, ei, return_net=True)
    R = (x.shape[0] + 127) // 128 * 128
    h = untile(net.debug_copy(3, (R * 128,), torch.float32).cpu().numpy(), x.shape[0], 128)
    net.close()
    _, _, st = O.forward(W, x, ei, cfg.n_iters, return_logits=True, return_states=True)
    assert np.abs(h - st["h"]).max() < 2e-3


def test_tiny_workload():
    w = S.WORKLOADS["tiny"]
    W = S.init_weights(w.model, w.weight_seed)
    x, ei = S.generate_event(w.event, w.seeds[0])
    s, rc = run_gpu(w.model, W, x, ei)
    assert rc == 0
    check_parity(s, W, x, ei, w.model.n_iters)


def test_mid_workload():
    w = S.WORKLOADS["mid"]
    W = S.init_weights(w.model, w.weight_seed)
    x, ei = S.generate_event(w.event, w.seeds[0])
    s, rc = run_gpu(w.model, W, x, ei)
    assert rc == 0
    check_parity(s, W, x, ei, w.model.n_iters)


def test_edge_cases_degenerate_graphs():
    cfg = S.ModelConfig(3, 2, 128, 2, 3)
    W = S.init_weights(cfg, 1)
    # single self-loop; duplicates; node with no edges
    x, _ = S.random_graph(4, 0, 3, 0)
    for ei in (np.array([[2], [2]], np.int32),
               np.array([[0, 0, 0, 1], [1, 1, 1, 1]], np.int32),
               np.array([[3, 1], [1, 3]], np.int32)):
        s, rc = run_gpu(cfg, W, x, ei)
        assert rc == 0
        check_parity(s, W, x, ei, cfg.n_iters)
    # duplicates score identically
    s, _ = run_gpu(cfg, W, x, np.array([[0, 0, 0, 1], [1, 1, 1, 1]], np.int32))
    assert s[0] == s[1] == s[2]


def test_hub_nodes_long_segments():
    """Two hubs: node 17 receives 60 % of the edges (one CSR segment across ~140 edge tiles) and
    the last node 20 % (the first node the aggregation blocks reach).  Long segments, sums that
    cross many tiles, and a CSR dominated by two keys; CSR bit-exact, scores against the oracle."""
    import torch
    n, e = 3000, 30000
    cfg = S.ModelConfig(3, 2, 128, 2, 3)
    W = S.init_weights(cfg, 5)
    x, ei = S.random_graph(n, e, 3, 21)
    k = np.random.default_rng(22).permutation(e)
    ei[1, k[:18000]] = 17
    ei[1, k[18000:24000]] = n - 1
    s, rc, net = run_gpu(cfg, W, x, ei, return_net=True)
    assert rc == 0
    rowptr, src_sorted, perm = O.csr_by_destination(ei[0], ei[1], n)
    np.testing.assert_array_equal(net.debug_copy(0, (n + 1,), torch.int32).cpu().numpy(), rowptr)
    np.testing.assert_array_equal(net.debug_copy(1, (e,), torch.int32).cpu().numpy(), perm)
    net.close()
    assert rowptr[18] - rowptr[17] >= 18000 and rowptr[n] - rowptr[n - 1] >= 6000
    check_parity(s, W, x, ei, cfg.n_iters)


def test_empty_edge_list_is_noop():
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    cfg = S.ModelConfig(3, 2, 64, 2, 2)
    net = InteractionNetwork(cfg, S.pack_blob(cfg, S.init_weights(cfg, 0)))
    out = net.infer(torch.zeros((5, 3), device="cuda"), torch.zeros((2, 0), dtype=torch.int32, device="cuda"))
    assert out.numel() == 0 and net.status() == 0
    net.close()


def test_out_of_range_index_reports_and_nans():
    cfg = S.ModelConfig(3, 2, 64, 2, 2)
    W = S.init_weights(cfg, 0)
    x, ei = S.random_graph(50, 300, 3, 9)
    bad = ei.copy()
    bad[1, 7] = 50          # dst out of range
    bad[0, 11] = -3         # src out of range
    s, rc = run_gpu(cfg, W, x, bad)
    assert rc == -5
    assert np.isnan(s[7]) and np.isnan(s[11])
    keep = np.ones(300, bool); keep[[7, 11]] = False
    check_parity(s[keep], W, x, bad[:, keep], cfg.n_iters)


def test_deterministic_and_batch_invariant():
    cfg = S.ModelConfig(12, 2, 128, 2, 3)
    W = S.init_weights(cfg, 4)
    spec = S.EventSpec(3000, 9, "powerlaw", 0.02, n_edges=9001)
    xb, eib = S.generate_batch(spec, (0, 1, 2))
    s1, _ = run_gpu(cfg, W, xb, eib)
    s2, _ = run_gpu(cfg, W, xb, eib)
    assert s1.tobytes() == s2.tobytes()
    parts = np.concatenate([run_gpu(cfg, W, *S.generate_event(spec, k))[0] for k in (0, 1, 2)])
    assert s1.tobytes() == parts.tobytes()
