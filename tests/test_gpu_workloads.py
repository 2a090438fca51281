"""GPU parity at the benchmark's sizes and on the remaining API paths (through the C ABI).

* full event (300k nodes, 1M edges, 12 features, H=128, T=8): every logit against the fp64 oracle;
* 16-event batch (4.8M nodes, 16M edges): a property that holds at any size -- the scores of an
  event inside the block-diagonal batch equal, bitwise, its scores when scored alone -- plus
  oracle parity of a 4-event batch at 1/10 scale;
* host-buffer entry point, profiling counters, workspace growth, H=64 with 3-layer MLPs."""
import numpy as np
import pytest

from oracle import gnn_oracle as O
from paper_2402_09633_gb300 import synthetic as S
from tests.gpu_util import check_parity, run_gpu

pytestmark = pytest.mark.gpu


def test_full_event_parity_against_oracle():
    w = S.WORKLOADS["full"]
    W = S.init_weights(w.model, w.weight_seed)
    x, ei = S.generate_event(w.event, 0)
    s, rc = run_gpu(w.model, W, x, ei)
    assert rc == 0
    err = check_parity(s, W, x, ei, w.model.n_iters)
    print(f"full event max logit error {err:.3e}")


def test_batch16_events_equal_their_standalone_scores():
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    w = S.WORKLOADS["batch16"]
    W = S.init_weights(w.model, w.weight_seed)
    xb, eib = S.generate_batch(w.event, w.seeds)
    assert xb.shape[0] == 4_800_000 and eib.shape[1] == 16_000_000
    net = InteractionNetwork(w.model, S.pack_blob(w.model, W))
    sb = net.infer(torch.from_numpy(xb).cuda(), torch.from_numpy(eib).cuda()).cpu().numpy()
    assert net.status() == 0
    E = w.event.n_edges
    for k in (0, 7, 15):
        x, ei = S.generate_event(w.event, w.seeds[k])
        s = net.infer(torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda()).cpu().numpy()
        assert s.tobytes() == sb[k * E:(k + 1) * E].tobytes(), f"event {k} differs inside the batch"
    net.close()


def test_64_copies_interleaved_equal_standalone():
    """Size well beyond the 16-event batch: 64 copies of the full event as one block-diagonal graph
    (19.2M nodes, 64M edges, about 75 GB of state), their edges interleaved in blocks of 1000 by a
    seeded random merge that keeps each copy's own edge order.  The CSR sort is stable, so every node
    sums its messages in the same order as in the standalone event: each copy's scores equal the
    standalone scores bit for bit."""
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    w = S.WORKLOADS["full"]
    W = S.init_weights(w.model, 0)
    x, ei = S.generate_event(w.event, 0)
    N, E, C, B = x.shape[0], ei.shape[1], 64, 1000
    assert E % B == 0
    labels = np.repeat(np.arange(C, dtype=np.int32), E // B)
    np.random.default_rng(5).shuffle(labels)
    blocks = np.argsort(labels, kind="stable").reshape(C, E // B)   # copy k's blocks land there, in order
    slots = (blocks[:, :, None] * B + np.arange(B)).reshape(C, E)    # slots[k] = where copy k's edges go
    eib = np.empty((2, C * E // B, B), np.int32)
    for k in range(C):
        eib[:, blocks[k], :] = (ei + np.int32(k * N)).reshape(2, E // B, B)
    eib = eib.reshape(2, C * E)
    xb = np.tile(x, (C, 1))
    net = InteractionNetwork(w.model, S.pack_blob(w.model, W))
    s1 = net.infer(torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda()).cpu().numpy()
    sb = net.infer(torch.from_numpy(xb).cuda(), torch.from_numpy(eib).cuda()).cpu().numpy()
    assert net.status() == 0
    net.close()
    for k in (0, 1, 31, 63):
        assert sb[slots[k]].tobytes() == s1.tobytes(), f"copy {k} differs inside the batch"
    assert np.array_equal(sb[slots].reshape(C, E), np.broadcast_to(s1, (C, E)))


def test_small_batch_parity_against_oracle():
    w = S.WORKLOADS["full"]
    W = S.init_weights(w.model, 0)
    spec = S.EventSpec(30000, 9, "powerlaw", 0.02, n_edges=100000)
    xb, eib = S.generate_batch(spec, (0, 1, 2, 3))
    s, rc = run_gpu(w.model, W, xb, eib)
    assert rc == 0
    check_parity(s, W, xb, eib, w.model.n_iters)


def test_host_entry_point_matches_device_path():
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    cfg = S.ModelConfig(12, 2, 128, 3, 3)
    W = S.init_weights(cfg, 2)
    x, ei = S.generate_event(S.EventSpec(5000, 9, "powerlaw", 0.02, n_edges=17000), 5)
    net = InteractionNetwork(cfg, S.pack_blob(cfg, W))
    dev = net.infer(torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda()).cpu().numpy()
    host = np.empty(ei.shape[1], np.float32)
    assert net.infer_host(x, ei, host) == 0                       # pageable numpy buffers
    assert host.tobytes() == dev.tobytes()
    xp, ep = torch.from_numpy(x).pin_memory(), torch.from_numpy(ei).pin_memory()
    sp = torch.empty(ei.shape[1], dtype=torch.float32).pin_memory()
    assert net.infer_host(xp, ep, sp) == 0                        # pinned tensors
    assert sp.numpy().tobytes() == dev.tobytes()
    bad = ei.copy(); bad[0, 3] = 10 ** 6
    assert net.infer_host(x, bad, host) == -5 and np.isnan(host[3])
    net.close()


def test_profile_counters_and_workspace_growth():
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    cfg = S.ModelConfig(3, 2, 128, 2, 3)
    W = S.init_weights(cfg, 0)
    net = InteractionNetwork(cfg, S.pack_blob(cfg, W))
    net.profile(True)
    for n, e in ((500, 1500), (4000, 12000)):                     # the second call grows the workspace
        x, ei = S.random_graph(n, e, 3, seed=n)
        s = net.infer(torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda()).cpu().numpy()
        check_parity(s, W, x, ei, cfg.n_iters)
    prof = net.profile_read()
    T = cfg.n_iters
    assert prof["edge_update"][1] == 2 * T and prof["node_update"][1] == 2 * T
    assert prof["aggregate"][1] == 2 * T and prof["classifier"][1] == 2
    assert prof["node_encoder"][1] == 2 and prof["edge_encoder"][1] == 2
    assert all(ms >= 0 for ms, _ in prof.values())
    net.profile(False)
    net.close()


@pytest.mark.parametrize("T,L", [(0, 3), (2, 3), (1, 4)])
def test_other_shapes(T, L):
    for H in (64, 128):
        cfg = S.ModelConfig(5, 2, H, T, L)
        W = S.init_weights(cfg, 3 + T + L)
        x, ei = S.random_graph(700, 2500, 5, seed=H + T)
        s, rc = run_gpu(cfg, W, x, ei)
        assert rc == 0
        check_parity(s, W, x, ei, T)
