"""Serving-style use of the C ABI (the paper's throughput levers: several model instances on one
GPU, Section 3.2): a gnn_infer call captured once into a CUDA graph and replayed, and several
contexts scoring different events concurrently on their own streams."""
import numpy as np
import pytest

from paper_2402_09633_gb300 import synthetic as S
from tests.gpu_util import check_parity

pytestmark = pytest.mark.gpu


def _event(seed, n=3000, e=10007):
    return S.generate_event(S.EventSpec(n, 9, "powerlaw", 0.02, n_edges=e), seed)


def test_cuda_graph_capture_and_replay():
    """After gnn_reserve, gnn_infer only enqueues kernels: it can be captured into a CUDA graph,
    and replaying the graph on new inputs (same sizes) gives the eager result bit for bit."""
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    cfg = S.ModelConfig(12, 2, 128, 3, 3)
    W = S.init_weights(cfg, 5)
    net = InteractionNetwork(cfg, S.pack_blob(cfg, W))
    x0, e0 = _event(0)
    x1, e1 = _event(1)
    assert x0.shape == x1.shape and e0.shape == e1.shape
    net.reserve(x0.shape[0], e0.shape[1])
    xs = torch.from_numpy(x0).cuda()
    es = torch.from_numpy(e0).cuda()
    out = torch.empty(e0.shape[1], dtype=torch.float32, device="cuda")
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        net.infer(xs, es, out, stream=stream)                 # warm-up outside capture
    stream.synchronize()
    eager0 = out.cpu().numpy().copy()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        net.infer(xs, es, out, stream=stream)
    for x, e, want in ((x1, e1, None), (x0, e0, eager0)):
        xs.copy_(torch.from_numpy(x)); es.copy_(torch.from_numpy(e))
        g.replay()
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        if want is not None:
            assert got.tobytes() == want.tobytes()
        else:
            eager = net.infer(torch.from_numpy(x).cuda(), torch.from_numpy(e).cuda()).cpu().numpy()
            assert got.tobytes() == eager.tobytes()
            check_parity(got, W, x, e, cfg.n_iters)
    assert net.status() == 0
    net.close()


def test_concurrent_contexts_on_separate_streams():
    """Several contexts (model instances) score different events on their own streams at the same
    time; each result equals its event scored alone."""
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    cfg = S.ModelConfig(12, 2, 128, 2, 3)
    W = S.init_weights(cfg, 6)
    events = [_event(k, n=2000 + 500 * k, e=7000 + 1000 * k) for k in range(3)]
    nets = [InteractionNetwork(cfg, S.pack_blob(cfg, W)) for _ in events]
    streams = [torch.cuda.Stream() for _ in events]
    inputs = [(torch.from_numpy(x).cuda(), torch.from_numpy(e).cuda()) for x, e in events]
    outs = []
    torch.cuda.synchronize()
    for net, st, (xs, es) in zip(nets, streams, inputs):
        with torch.cuda.stream(st):
            outs.append(net.infer(xs, es, stream=st))
    for net, st in zip(nets, streams):
        assert net.status(stream=st) == 0
    ref = InteractionNetwork(cfg, S.pack_blob(cfg, W))
    for (x, e), (xs, es), o in zip(events, inputs, outs):
        alone = ref.infer(xs, es).cpu().numpy()
        assert o.cpu().numpy().tobytes() == alone.tobytes()
        check_parity(alone, W, x, e, cfg.n_iters)
    ref.close()
    for net in nets:
        net.close()
