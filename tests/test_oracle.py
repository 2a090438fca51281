"""Pins of the fp64 oracle against facts fixed by mathematics, not by itself.

Each check targets a plausible mistake: a dropped term (bias, gamma, beta, the
edge-state block), a wrong sign or index (source/destination swap, wrap
direction, aggregation at the source), a transposed operand, or an
iteration that forgets to carry the edge state."""
import math

import numpy as np
import pytest

from oracle import gnn_oracle as O
from paper_2402_09633_gb300 import synthetic as S

EPS = 1e-5


# ----------------------------------------------------------------- primitives

def test_layer_norm_closed_forms():
    g = np.array([1.0, 1.0, 1.0, 1.0]); b = np.zeros(4)
    # [1,2,3,4]: mean 2.5, biased variance 1.25
    v = np.array([1.0, 2.0, 3.0, 4.0])
    want = (v - 2.5) / math.sqrt(1.25 + EPS)
    np.testing.assert_allclose(O.layer_norm(v, g, b, EPS), want, rtol=0, atol=1e-15)
    # affine part: gamma scales, beta shifts, per feature
    g2 = np.array([2.0, -1.0, 0.5, 3.0]); b2 = np.array([0.1, 0.2, -0.3, 0.4])
    np.testing.assert_allclose(O.layer_norm(v, g2, b2, EPS), g2 * want + b2, atol=1e-15)
    # constant row: variance 0 -> output is beta exactly
    np.testing.assert_array_equal(O.layer_norm(np.full(4, 7.25), g2, b2, EPS), b2)
    # two features: (g1*d/s + b1, -g2*d/s + b2) with d = (v1 - v2)/2, s = sqrt(d^2 + eps)
    for v1, v2 in [(0.3, -0.1), (0.001, 0.0), (-5.0, 2.0)]:
        d = (v1 - v2) / 2; s = math.sqrt(d * d + EPS)
        got = O.layer_norm(np.array([v1, v2]), np.array([1.5, 0.5]), np.array([0.1, -0.2]), EPS)
        np.testing.assert_allclose(got, [1.5 * d / s + 0.1, -0.5 * d / s - 0.2], atol=1e-15)


def test_sigmoid_special_values():
    np.testing.assert_allclose(O.sigmoid(np.array([0.0])), [0.5], atol=0)
    np.testing.assert_allclose(O.sigmoid(np.array([math.log(3.0)])), [0.75], atol=1e-15)
    np.testing.assert_allclose(O.sigmoid(np.array([-math.log(3.0)])), [0.25], atol=1e-15)
    z = np.linspace(-30, 30, 61)
    np.testing.assert_allclose(O.sigmoid(z) + O.sigmoid(-z), 1.0, atol=1e-15)
    big = O.sigmoid(np.array([-800.0, 800.0]))          # no overflow, saturates
    assert big[0] == 0.0 and big[1] == 1.0


def test_mlp_single_layer_by_hand():
    # W [2,3] non-symmetric: a transposed operand cannot even be applied
    W = np.array([[1.0, -2.0, 0.5], [0.25, 1.0, -1.0]]); b = np.array([0.3, -0.2])
    g = np.array([2.0, 0.5]); be = np.array([-0.1, 0.05])
    x = np.array([0.4, 0.1, -0.6])
    v1 = 0.4 - 0.2 - 0.3 + 0.3          # = 0.2
    v2 = 0.1 + 0.1 + 0.6 - 0.2          # = 0.6
    d = (v1 - v2) / 2; s = math.sqrt(d * d + EPS)
    want = [max(2.0 * d / s - 0.1, 0.0), max(-0.5 * d / s + 0.05, 0.0)]
    np.testing.assert_allclose(O.mlp(x[None], [(W, b, g, be)], EPS)[0], want, atol=1e-15)
    assert want[0] == 0.0 and want[1] > 0.0            # ReLU clipped one feature


def test_edge_features_wrap_and_sign():
    x = np.array([[0.1, 0.0], [0.3, 0.5], [0.2, 0.9], [0.4, -0.8], [0.5, -0.5]], np.float32)
    src = np.array([0, 1, 2, 3, 2, 4, 0])
    dst = np.array([1, 2, 3, 2, 4, 2, 0])
    f = O.edge_features(x, src, dst)
    f32 = np.float32
    want_dr = [f32(0.3) - f32(0.1), f32(0.2) - f32(0.3), f32(0.4) - f32(0.2), f32(0.2) - f32(0.4),
               f32(0.5) - f32(0.2), f32(0.2) - f32(0.5), f32(0.0)]
    # dphi = phi_dst - phi_src wrapped into (-1, 1]
    want_dp = [f32(0.5), f32(0.9) - f32(0.5), (f32(-0.8) - f32(0.9)) + f32(2.0),
               (f32(0.9) - f32(-0.8)) - f32(2.0), f32(-0.5) - f32(0.9) + f32(2.0),
               (f32(0.9) - f32(-0.5)) - f32(2.0), f32(0.0)]
    np.testing.assert_array_equal(f[:, 0], np.array(want_dr, np.float32))
    np.testing.assert_array_equal(f[:, 1], np.array(want_dp, np.float32))
    assert f.dtype == np.float32
    # exact boundaries: +1 stays, -1 maps to +1, +-2 edge cases stay in (-1, 1]
    w = O.wrap_dphi_f32(np.array([1.0, -1.0, 1.5, -1.5, 0.0, -0.999], np.float32))
    np.testing.assert_array_equal(w, np.array([1.0, 1.0, -0.5, 0.5, 0.0, -0.999], np.float32))


def test_csr_against_brute_force():
    rng = np.random.default_rng(3)
    for n, e in [(1, 5), (7, 0), (9, 40), (33, 200)]:
        src = rng.integers(0, n, e); dst = rng.integers(0, n, e)
        rowptr, src_sorted, perm = O.csr_by_destination(src, dst, n)
        # brute force: scan nodes in order, then edges in input order
        want_perm = [k for j in range(n) for k in range(e) if dst[k] == j]
        assert perm.tolist() == want_perm
        assert src_sorted.tolist() == [int(src[k]) for k in want_perm]
        want_rowptr = [0]
        for j in range(n):
            want_rowptr.append(want_rowptr[-1] + sum(1 for k in range(e) if dst[k] == j))
        assert rowptr.tolist() == want_rowptr


def test_aggregation_equals_dense_incidence_product():
    rng = np.random.default_rng(5)
    for n, e in [(1, 3), (8, 30), (64, 500)]:
        dst = rng.integers(0, n, e)
        m = rng.standard_normal((e, 6))
        D = np.zeros((n, e)); D[dst, np.arange(e)] = 1.0     # D[j, k] = [dst(k) = j]
        np.testing.assert_allclose(O.aggregate(m, dst, n), D @ m, rtol=0, atol=1e-12)
    # a node without in-edges aggregates to zero
    a = O.aggregate(np.ones((2, 3)), np.array([0, 0]), 3)
    np.testing.assert_array_equal(a[1:], 0.0)


# ----------------------------------------------------------- worked example

HAND_EPS = 1.0   # large eps keeps the 2-feature LayerNorm out of its +-1 saturation


def _ln2(v1, v2, g, b):
    """LayerNorm of a 2-vector: only d = (v1 - v2)/2 matters."""
    d = (v1 - v2) / 2.0
    s = math.sqrt(d * d + HAND_EPS)
    return (g[0] * d / s + b[0], -g[1] * d / s + b[1])


def _relu2(p):
    return (max(p[0], 0.0), max(p[1], 0.0))


def _hand_model():
    """H = 2, one layer per MLP, T = 1 (and T = 2), all weights small and asymmetric."""
    one, zero = np.ones(2), np.zeros(2)
    Wn = np.array([[0.0, 1.0], [0.0, -1.0]]); bn = np.zeros(2)                 # node encoder
    We = np.array([[1.0, 1.0], [0.0, 0.0]]); be_ = np.array([-0.45, 0.0])     # edge encoder
    # edge network on [h_src(2), h_dst(2), e(2)]
    Wm = np.array([[0.7, -1.1, 0.3, 0.9, -0.6, 1.3], [0.2, 0.4, -0.5, 0.1, 0.8, -0.2]])
    bm = np.array([0.05, -0.1])
    gm = np.array([1.2, 0.8]); btm = np.array([0.1, -0.05])
    # node network on [h(2), a(2)]
    Wu = np.array([[0.5, -0.3, 0.9, -0.7], [-0.4, 0.6, 0.2, 0.35]])
    bu = np.array([-0.02, 0.03])
    gu = np.array([0.9, 1.1]); btu = np.array([-0.04, 0.02])
    # classifier on [h_src, h_dst, e]
    Wc = np.array([[-0.8, 0.6, 1.0, -0.2, 0.45, -0.9], [0.3, -0.7, 0.25, 0.5, -0.35, 0.6]])
    bc = np.array([0.08, -0.03])
    gc = np.array([1.05, 0.95]); btc = np.array([0.02, 0.07])
    W = {"node_encoder": [(Wn, bn, one, zero)], "edge_encoder": [(We, be_, one, zero)],
         "edge_network": [(Wm, bm, gm, btm)], "node_network": [(Wu, bu, gu, btu)],
         "edge_classifier": [(Wc, bc, gc, btc)],
         "head_w": np.array([1.5, -2.0]), "head_b": np.array([0.25])}
    return W


def _hand_forward(W, x, src, dst, T, rnd=None):
    """Scalar forward of the hand model; `rnd` (if given) rounds every layer output and the
    aggregate, as the bf16 model does."""
    f32 = np.float32
    n, E = x.shape[0], len(src)
    r = rnd if rnd is not None else (lambda t: t)

    def lin(Wb, z):
        Wm, b = Wb
        return [sum(Wm[r][c] * z[c] for c in range(len(z))) + b[r] for r in range(2)]

    def layer(params, z):
        Wm, b, g, bt = params[0]
        v = lin((Wm, b), z)
        o = _relu2(_ln2(v[0], v[1], g, bt))
        return (r(o[0]), r(o[1]))

    h = [layer(W["node_encoder"], [float(x[j][0]), float(x[j][1])]) for j in range(n)]
    e = []
    for k in range(E):
        i, j = src[k], dst[k]
        dr = float(f32(x[j][0]) - f32(x[i][0]))
        dp = f32(x[j][1]) - f32(x[i][1])
        dp = float(dp - f32(2) if dp > 1 else (dp + f32(2) if dp <= -1 else dp))
        e.append(layer(W["edge_encoder"], [dr, dp]))
    for _ in range(T):
        m = [layer(W["edge_network"], list(h[src[k]]) + list(h[dst[k]]) + list(e[k])) for k in range(E)]
        e = m
        a = [[0.0, 0.0] for _ in range(n)]
        for k in range(E):
            a[dst[k]][0] += m[k][0]; a[dst[k]][1] += m[k][1]
        a = [[r(a[j][0]), r(a[j][1])] for j in range(n)]
        h = [layer(W["node_network"], list(h[j]) + a[j]) for j in range(n)]
    logits = []
    for k in range(E):
        c = layer(W["edge_classifier"], list(h[src[k]]) + list(h[dst[k]]) + list(e[k]))
        logits.append(W["head_w"][0] * c[0] + W["head_w"][1] * c[1] + W["head_b"][0])
    return logits


HAND_X = np.array([[0.1, 0.0], [0.2, 0.5], [0.3, 0.9], [0.4, -0.8]], np.float32)
HAND_EI = np.array([[0, 1, 0, 2], [1, 2, 2, 3]], np.int32)


@pytest.mark.parametrize("T", [1, 2])
def test_worked_example_4_nodes_4_edges(T):
    W = _hand_model()
    _, logits = O.forward(W, HAND_X, HAND_EI, T, HAND_EPS, return_logits=True)
    want = _hand_forward(W, HAND_X, HAND_EI[0].tolist(), HAND_EI[1].tolist(), T)
    np.testing.assert_allclose(logits, want, rtol=0, atol=1e-12)
    # the wrap branch and both ReLU branches are exercised; node 0 has no in-edge
    assert np.abs(np.diff(logits)).min() > 1e-3


def test_worked_example_detects_wiring_mistakes():
    """The worked example separates the right wiring from plausible wrong ones."""
    W = _hand_model()
    want = np.array(_hand_forward(W, HAND_X, [0, 1, 0, 2], [1, 2, 2, 3], 1))
    # source/destination swapped everywhere
    swapped = np.array(_hand_forward(W, HAND_X, [1, 2, 2, 3], [0, 1, 0, 2], 1))
    assert np.abs(swapped - want).max() > 1e-3
    # zeroing the edge-state block of the edge network changes the answer
    W2 = _hand_model(); Wm, bm, gm, btm = W2["edge_network"][0]
    Wm = Wm.copy(); Wm[:, 4:] = 0.0; W2["edge_network"] = [(Wm, bm, gm, btm)]
    assert np.abs(np.array(O.forward(W2, HAND_X, HAND_EI, 1, HAND_EPS, return_logits=True)[1]) - want).max() > 1e-3


# --------------------------------------------------------------- invariances

def _small_model(H=8, L=2, Fn=3, seed=1):
    cfg = S.ModelConfig(Fn, 2, H, 2, L)
    return cfg, S.init_weights(cfg, seed)


def test_node_relabelling_invariance():
    cfg, W = _small_model()
    x, ei = S.random_graph(40, 150, 3, seed=7)
    s0 = O.forward(W, x, ei, cfg.n_iters)
    p = np.random.default_rng(0).permutation(40)          # new id of old node k is p[k]
    x2 = np.empty_like(x); x2[p] = x
    ei2 = p[ei].astype(np.int32)
    s1 = O.forward(W, x2, ei2, cfg.n_iters)
    np.testing.assert_allclose(s1, s0, rtol=0, atol=1e-13)


def test_edge_reordering_equivariance():
    cfg, W = _small_model()
    x, ei = S.random_graph(40, 150, 3, seed=8)
    s0 = O.forward(W, x, ei, cfg.n_iters)
    q = np.random.default_rng(1).permutation(150)
    s1 = O.forward(W, x, ei[:, q], cfg.n_iters)
    np.testing.assert_allclose(s1, s0[q], rtol=0, atol=1e-12)


def test_block_diagonal_batch_is_concatenation():
    cfg, W = _small_model()
    spec = S.EventSpec(200, 0, "fanout", 0.5)
    xs, eis = [], []
    for s in (0, 1, 2):
        x, ei = S.generate_event(spec, s); xs.append(x); eis.append(ei)
    xb, eib = S.generate_batch(spec, (0, 1, 2))
    sb = O.forward(W, xb, eib, cfg.n_iters)
    parts = np.concatenate([O.forward(W, x, ei, cfg.n_iters) for x, ei in zip(xs, eis)])
    np.testing.assert_allclose(sb, parts, rtol=0, atol=1e-12)


def test_duplicate_edge_doubles_its_message():
    """A duplicated edge contributes its message twice to its destination."""
    cfg, W = _small_model()
    x, ei = S.random_graph(10, 20, 3, seed=9)
    ei2 = np.concatenate([ei, ei[:, :1]], axis=1)
    f = O.edge_features(x, ei2[0], ei2[1]).astype(np.float64)
    e0 = O.mlp(f, W["edge_encoder"], EPS)
    h0 = O.mlp(x.astype(np.float64), W["node_encoder"], EPS)
    m = O.mlp(np.concatenate([h0[ei2[0]], h0[ei2[1]], e0], 1), W["edge_network"], EPS)
    a1 = O.aggregate(m[:-1], ei2[1, :-1], 10)
    a2 = O.aggregate(m, ei2[1], 10)
    j = ei[1, 0]
    np.testing.assert_allclose(a2[j] - a1[j], m[0], atol=1e-12)
    np.testing.assert_allclose(np.delete(a2 - a1, j, axis=0), 0.0, atol=0)
    # and the duplicate's own score equals the original's
    s = O.forward(W, x, ei2, cfg.n_iters)
    assert s[-1] == s[0]


def test_empty_graph_and_isolated_nodes():
    cfg, W = _small_model()
    x, _ = S.random_graph(5, 0, 3, seed=0)
    s = O.forward(W, x, np.zeros((2, 0), np.int32), cfg.n_iters)
    assert s.shape == (0,)
    # self-loop only
    s = O.forward(W, x, np.array([[2], [2]], np.int32), cfg.n_iters)
    assert s.shape == (1,) and 0.0 < s[0] < 1.0


def test_golden_regression():
    """Oracle output on a fixed seeded graph, written by tests/golden/make_golden.py."""
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "oracle_small_logits.txt")
    want = np.loadtxt(path)
    from tests.golden.make_golden import golden_case
    W, x, ei, T = golden_case()
    _, got = O.forward(W, x, ei, T, return_logits=True)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)


def _mutants():
    """Plausible mistakes, planted in the oracle (on the CPU) one at a time."""
    ln, agg, ef, relu, sig = O.layer_norm, O.aggregate, O.edge_features, O.relu, O.sigmoid

    def ln_no_beta(v, g, b, eps):
        return ln(v, g, 0 * b, eps)

    def ln_unbiased(v, g, b, eps):
        mu = v.mean(-1, keepdims=True)
        var = ((v - mu) ** 2).sum(-1, keepdims=True) / max(v.shape[-1] - 1, 1)
        return g * (v - mu) / np.sqrt(var + eps) + b

    def agg_twice(m, dst, n, dtype=np.float64):
        return 2 * agg(m, dst, n, dtype)

    def ef_neg(x, s, d):
        return -ef(x, s, d)

    def relu_none(v):
        return v

    return {"ln_no_beta": ("layer_norm", ln_no_beta), "ln_unbiased": ("layer_norm", ln_unbiased),
            "agg_twice": ("aggregate", agg_twice), "features_sign": ("edge_features", ef_neg),
            "no_relu": ("relu", relu_none)}


@pytest.mark.parametrize("name", sorted(_mutants()))
def test_worked_example_kills_planted_mistakes(name, monkeypatch):
    attr, fn = _mutants()[name]
    W = _hand_model()
    want = np.array(_hand_forward(W, HAND_X, HAND_EI[0].tolist(), HAND_EI[1].tolist(), 2))
    monkeypatch.setattr(O, attr, fn)
    _, got = O.forward(W, HAND_X, HAND_EI, 2, HAND_EPS, return_logits=True)
    assert np.abs(got - want).max() > 1e-6, name


# ------------------------------------------------------------- bf16 model

def _bf16_scalar(t: float) -> float:
    """Nearest bfloat16 of a Python float: t = m * 2**e with 0.5 <= |m| < 1, keep 8
    significant bits; Python's round() takes halfway cases to even."""
    if t == 0.0:
        return 0.0
    m, e = math.frexp(t)
    return math.ldexp(round(m * 256), e - 8)


def test_round_bf16_values():
    # spacing next to 1 is 2^-7; exact halfway cases go to the even neighbour
    cases = {1.0: 1.0, 1.0 + 2 ** -8: 1.0, 1.0 + 3 * 2 ** -8: 1.0 + 2 ** -6, 1.0 + 2 ** -7: 1.0 + 2 ** -7,
             0.1: 0.10009765625, -2.5: -2.5, 255.5: 256.0, 257.0: 256.0, 3.0e-3: 0.0030059814453125}
    got = O.round_bf16(np.array(list(cases)))
    np.testing.assert_array_equal(got, list(cases.values()))
    # agrees with an independent bit-level rounding of float32 values
    v = np.random.default_rng(3).standard_normal(20000).astype(np.float32) * 7
    np.testing.assert_array_equal(O.round_bf16(v.astype(np.float64)), S._round_bf16(v).astype(np.float64))
    assert all(O.round_bf16(np.array([t]))[0] == _bf16_scalar(t) for t in v[:500].tolist())


@pytest.mark.parametrize("T", [1, 2])
def test_bf16_worked_example(T):
    """The bf16 model rounds every layer output and the aggregate, nothing else."""
    W = _hand_model()
    _, got = O.forward(W, HAND_X, HAND_EI, T, HAND_EPS, return_logits=True, bf16=True)
    want = _hand_forward(W, HAND_X, HAND_EI[0].tolist(), HAND_EI[1].tolist(), T, rnd=_bf16_scalar)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
    plain = _hand_forward(W, HAND_X, HAND_EI[0].tolist(), HAND_EI[1].tolist(), T)
    assert np.abs(np.array(want) - np.array(plain)).max() > 1e-4      # the rounding points are live


def test_bf16_model_close_to_unrounded_model():
    cfg = S.ModelConfig(3, 2, 64, 2, 2, S.PRECISION_BF16)
    W = S.init_weights(cfg, 4)
    x, ei = S.random_graph(60, 300, 3, 2)
    _, z64 = O.forward(W, x, ei, cfg.n_iters, return_logits=True)
    _, zb = O.forward(W, x, ei, cfg.n_iters, return_logits=True, bf16=True)
    d = np.abs(zb - z64)
    assert 1e-4 < d.max() < 0.5 and d.mean() < 0.05


# ------------------------------------------------------------- track labels

def _bfs_labels(edges, n):
    """Brute force: breadth-first search from every unvisited node in increasing id order."""
    adj = [[] for _ in range(n)]
    for a, b in edges:
        adj[a].append(b); adj[b].append(a)
    lab = [-1] * n
    for s0 in range(n):
        if lab[s0] >= 0:
            continue
        lab[s0] = s0
        todo = [s0]
        while todo:
            x = todo.pop()
            for y in adj[x]:
                if lab[y] < 0:
                    lab[y] = s0; todo.append(y)
    return lab


def test_track_labels_against_breadth_first_search():
    rng = np.random.default_rng(8)
    for n, m in [(1, 0), (5, 3), (40, 30), (300, 250), (300, 900)]:
        ei = rng.integers(0, n, size=(2, m)).astype(np.int32)
        sc = rng.random(m)
        for thr in (0.0, 0.5, 0.9):
            kept = [(int(a), int(b)) for a, b, x in zip(ei[0], ei[1], sc) if x > thr]
            assert O.track_labels(sc, ei, n, thr).tolist() == _bfs_labels(kept, n)


def test_track_labels_special_cases():
    ei = np.array([[0, 1, 3, 4, 2], [1, 2, 3, 9, 7]], np.int32)    # self-loop, out-of-range endpoints
    sc = np.array([0.9, 0.9, 0.9, 0.9, np.nan])
    assert O.track_labels(sc, ei, 6, 0.5).tolist() == [0, 0, 0, 3, 4, 5]
    assert O.track_labels(sc, ei, 6, 0.95).tolist() == [0, 1, 2, 3, 4, 5]   # nothing kept
    assert O.track_labels(np.zeros(0), np.zeros((2, 0), np.int32), 3).tolist() == [0, 1, 2]
    # a path given leaves-first still labels every hit with the smallest id
    ei = np.array([[5, 4, 3, 2, 1], [4, 3, 2, 1, 0]], np.int32)
    assert O.track_labels(np.ones(5), ei, 6).tolist() == [0] * 6


def test_track_labels_against_library_components():
    sp = pytest.importorskip("scipy.sparse")
    csg = pytest.importorskip("scipy.sparse.csgraph")
    rng = np.random.default_rng(9)
    n, m = 5000, 4000
    ei = rng.integers(0, n, size=(2, m)).astype(np.int32)
    sc = rng.random(m)
    keep = sc > 0.3
    g = sp.coo_matrix((np.ones(keep.sum()), (ei[0][keep], ei[1][keep])), shape=(n, n))
    _, comp = csg.connected_components(g, directed=True, connection="weak")
    smallest = np.full(comp.max() + 1, n)
    np.minimum.at(smallest, comp, np.arange(n))
    np.testing.assert_array_equal(O.track_labels(sc, ei, n, 0.3), smallest[comp])


# ------------------------------------------------------------- filtering

def test_filter_scores_by_hand():
    """One layer, H = 2, F_n = 1: s = sigmoid(w . ReLU(LN(W [x_src, x_dst] + b)) + b_o)."""
    fw = {"layers": [(np.array([[1.0, -2.0], [0.5, 1.5]]), np.array([0.1, -0.3]), np.array([2.0, 0.5]),
                      np.array([-0.1, 0.05]))],
          "head_w": np.array([1.5, -0.75]), "head_b": np.array([0.2])}
    x = np.array([[0.4], [-0.3], [0.9]], np.float32)
    ei = np.array([[0, 2, 1, 0], [1, 0, 2, 5]], np.int32)            # the last edge is out of range
    got_s, got_z = O.filter_scores(fw, x, ei, HAND_EPS, return_logits=True)
    for k in range(3):
        a, b = float(x[ei[0, k], 0]), float(x[ei[1, k], 0])
        v1, v2 = a - 2.0 * b + 0.1, 0.5 * a + 1.5 * b - 0.3
        h = _relu2(_ln2(v1, v2, (2.0, 0.5), (-0.1, 0.05)))
        z = 1.5 * h[0] - 0.75 * h[1] + 0.2
        assert abs(got_z[k] - z) < 1e-12 and abs(got_s[k] - 1.0 / (1.0 + math.exp(-z))) < 1e-12
    assert np.isnan(got_s[3]) and np.isnan(got_z[3])
    # swapping source and destination changes the score (the input is ordered [x_src, x_dst])
    assert abs(O.filter_scores(fw, x, ei[::-1, :1], HAND_EPS)[0] - got_s[0]) > 1e-3


def test_apply_filtering_keeps_order_and_drops_nan():
    ei = np.array([[0, 1, 2, 3, 4], [5, 6, 7, 8, 9]], np.int32)
    sc = np.array([0.9, 0.2, np.nan, 0.51, 0.5])
    kept, ids = O.apply_filtering(sc, ei, 0.5)
    assert ids.tolist() == [0, 3]
    assert kept.tolist() == [[0, 3], [5, 8]]


# ------------------------------------------------------------- embedding and graph building

def test_embed_is_unit_length_and_matches_hand_layer():
    ew = {"layers": [(np.array([[1.0, -0.5], [0.25, 2.0]]), np.array([0.1, 0.0]), np.array([1.0, 1.0]),
                      np.array([0.0, 0.3]))],
          "out_w": np.array([[1.0, 2.0], [-1.0, 0.5], [0.0, 1.0]]), "out_b": np.array([0.1, 0.0, -0.2])}
    x = np.array([[0.3, 0.7], [-1.0, 0.2]], np.float32)
    y = O.embed(ew, x, HAND_EPS)
    for k in range(2):
        a, b = float(x[k, 0]), float(x[k, 1])
        h = _relu2(_ln2(a - 0.5 * b + 0.1, 0.25 * a + 2.0 * b, (1.0, 1.0), (0.0, 0.3)))
        z = np.array([h[0] + 2 * h[1] + 0.1, -h[0] + 0.5 * h[1], h[1] - 0.2])
        np.testing.assert_allclose(y[k], z / np.linalg.norm(z), atol=1e-12)
    np.testing.assert_allclose(np.linalg.norm(y, axis=1), 1.0, atol=1e-12)


def test_radius_graph_against_brute_force_and_kdtree():
    rng = np.random.default_rng(11)
    emb = rng.standard_normal((400, 5)).astype(np.float32)
    emb /= np.linalg.norm(emb, axis=1, keepdims=True)
    r_col = rng.integers(0, 4, 400).astype(np.float32)          # layer-like radii with many ties
    radius = 0.45
    got = O.radius_graph(emb, r_col, radius)
    want = []
    for i in range(400):                                         # float64 brute force, away from the boundary
        for j in range(i + 1, 400):
            d2 = float(((emb[i].astype(np.float64) - emb[j]) ** 2).sum())
            if d2 < radius * radius:
                a, b = (i, j) if (r_col[i] < r_col[j] or (r_col[i] == r_col[j] and i < j)) else (j, i)
                want.append((a, b))
    assert len(want) > 200
    got_set, want_set = set(map(tuple, got.tolist())), set(want)
    diff = got_set ^ want_set
    for a, b in diff:                                            # only pairs on the boundary may differ
        d2 = float(((emb[a].astype(np.float64) - emb[b]) ** 2).sum())
        assert abs(d2 - radius * radius) < 1e-5
    kd = pytest.importorskip("scipy.spatial")
    cand = np.array(sorted(kd.cKDTree(emb.astype(np.float64)).query_pairs(radius * 1.001)), np.int64)
    np.testing.assert_array_equal(O.radius_graph(emb, r_col, radius, cand), got)
