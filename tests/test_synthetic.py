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


def test_full_event_structure():
    """The 300k-hit / 1M-edge event of the headline benchmark: exact edge count, power-law
    in-degree capped at 40 with nothing into layer 0, sources on the previous layer, distinct
    sources per hit, and the |dphi| window (widened only where a hit needs more candidates)."""
    x, ei = S.generate_event(S.WORKLOADS["full"].event, 0)
    assert x.shape == (300000, 12) and ei.shape == (2, 1000000) and ei.dtype == np.int32
    src, dst = ei.astype(np.int64)
    layer = np.searchsorted(np.asarray(S.LAYER_RADII_MM, int), np.round(x[:, 0] * 1000).astype(int))
    assert np.all(layer[src] == layer[dst] - 1)
    deg = np.bincount(dst, minlength=300000)
    assert deg.max() <= S.MAX_IN_DEGREE and deg[layer == 0].sum() == 0
    assert np.unique(src * 300000 + dst).size == 1000000           # no duplicate edge
    dphi = np.abs(np.angle(np.exp(1j * np.pi * (x[dst, 1].astype(np.float64) - x[src, 1]))))
    assert np.mean(dphi < 0.02) > 0.999
    hist = np.bincount(deg[layer > 0], minlength=S.MAX_IN_DEGREE + 1)
    assert hist[0] > hist[5] > hist[20] > 0                         # a decreasing heavy tail


def test_filter_and_embed_blob_layouts():
    cfg = S.ModelConfig(12, 2, 128, 8, 3)
    fw = S.init_filter_weights(cfg, 1)
    fb = S.pack_filter_blob(cfg, fw)
    hdr = np.frombuffer(fb[:32], "<i4")
    assert hdr[0] == S.FILTER_MAGIC and hdr[2] == 12 and hdr[3] == 128 and hdr[4] == 3
    n = int(np.frombuffer(fb[40:48], "<i8")[0])
    assert n == 128 * 24 + 3 * 128 + 2 * (128 * 128 + 3 * 128) + 128 + 1
    assert len(fb) == S.BLOB_HEADER_BYTES + 4 * n
    ew = S.init_embed_weights(cfg, 8, 2)
    eb = S.pack_embed_blob(cfg, ew)
    hdr = np.frombuffer(eb[:32], "<i4")
    assert hdr[0] == S.EMBED_MAGIC and hdr[6] == 8
    n = int(np.frombuffer(eb[40:48], "<i8")[0])
    assert n == 128 * 12 + 3 * 128 + 2 * (128 * 128 + 3 * 128) + 8 * 128 + 8
    f = np.frombuffer(eb[S.BLOB_HEADER_BYTES:], "<f4")
    np.testing.assert_array_equal(f[-8:], ew["out_b"])
