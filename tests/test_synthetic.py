"""Seeded input generator: determinism, shapes, and the structure of the events."""
import numpy as np

from paper_2402_09633_gb300 import synthetic as S


def test_same_seed_same_bytes():
    spec = S.EventSpec(3000, 9, "powerlaw", 0.02, n_edges=10000)
    a = S.generate_event(spec, 4); b = S.generate_event(spec, 4)
    assert a[0].tobytes() == b[0].tobytes() and a[1].tobytes() == b[1].tobytes()
    c = S.generate_event(spec, 5)
    assert a[1].tobytes() != c[1].tobytes()


def test_fanout_event_structure():
    spec = S.WORKLOADS["tiny"].event
    x, ei = S.generate_event(spec, 0)
    assert x.shape == (2000, 3) and x.dtype == np.float32 and ei.dtype == np.int32
    layer = np.round(x[:, 0] * 1000).astype(int)
    radii = np.asarray(S.LAYER_RADII_MM, int)
    li = np.searchsorted(radii, layer)
    src, dst = ei
    assert np.all(li[dst] == li[src] + 1)                  # next-layer links only
    dphi = np.abs(np.angle(np.exp(1j * np.pi * (x[dst, 1].astype(np.float64) - x[src, 1]))))
    assert dphi.max() < 0.3 + 1e-6
    out_deg = np.bincount(src, minlength=2000)
    assert out_deg.max() <= 4 and 7000 <= ei.shape[1] <= 8000
    assert len({(a, b) for a, b in zip(src, dst)}) == ei.shape[1]   # distinct targets


def test_powerlaw_event_structure():
    spec = S.EventSpec(30000, 9, "powerlaw", 0.02, n_edges=100000)
    x, ei = S.generate_event(spec, 0)
    assert x.shape == (30000, 12) and ei.shape == (2, 100000)
    deg = np.bincount(ei[1], minlength=30000)
    assert deg.max() <= S.MAX_IN_DEGREE and deg[:3000].sum() == 0
    assert abs(deg[3000:].mean() - 100000 / 27000) < 1e-9
    assert (np.sort(ei[1]) != ei[1]).any()                  # shuffled order


def test_blob_layout():
    cfg = S.ModelConfig(12, 2, 128, 8, 3)
    W = S.init_weights(cfg, 0)
    blob = S.pack_blob(cfg, W)
    assert len(blob) == S.BLOB_HEADER_BYTES + 4 * S.blob_n_floats(cfg)
    f = np.frombuffer(blob[S.BLOB_HEADER_BYTES:], "<f4")
    np.testing.assert_array_equal(f[:128 * 12], W["node_encoder"][0][0].ravel())
    np.testing.assert_array_equal(f[-129:-1], W["head_w"])


def test_bf16_weights_are_bf16_numbers():
    cfg = S.ModelConfig(12, 2, 128, 8, 3, S.PRECISION_BF16)
    W = S.init_weights(cfg, 0)
    u = W["edge_network"][0][0].view(np.uint32)
    assert np.all((u & 0xFFFF) == 0)
