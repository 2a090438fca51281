"""Oracle: plain, slow, fp64 CPU evaluation of the interaction-network edge classifier.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this module:
only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may call it.  It shares no code with the CUDA path.

What it computes (Section 2.1: space points in, candidate edges between them,
the edge-classification step is an interaction network whose per-edge scores
feed the connected-components step).  The paper cites the interaction network
without writing out its equations, so the network below is the plain
message-passing definition the benchmark specifies, evaluated in float64:

    MLP(v)      = for each layer l: v <- ReLU(LayerNorm_l(W_l v + b_l))
    LayerNorm   : mean and biased variance over the H features,
                  gamma * (v - mean) / sqrt(var + eps) + beta
    f_ij        = (x_j[0] - x_i[0], wrap(x_j[1] - x_i[1]))   for edge i -> j
    h_j         = MLP_node_encoder(x_j);  e_ij = MLP_edge_encoder(f_ij)
    repeat T times:
        m_ij    = MLP_edge_network([h_i, h_j, e_ij]);  e_ij <- m_ij
        a_j     = sum over edges (i -> j) of m_ij     (zero when j has no in-edge)
        h_j     = MLP_node_network([h_j, a_j])
    logit_ij    = w_o . MLP_edge_classifier([h_i, h_j, e_ij]) + b_o
    score_ij    = 1 / (1 + exp(-logit_ij))

Edge features use the input's precision: the phi difference of two float32
features is rounded to float32 and the wrap into (-1, 1] (units of pi; exact
+-1 maps to +1) is decided on that float32 value, so the oracle and a float32
kernel take the same wrap decision.

The bf16 model (bf16 weights and activations, wider accumulation) is the same
network with every activation rounded to the nearest bfloat16 (ties to even):
the output of every MLP layer (so every input of a Linear layer after the
first, and the stored states h and e) and the aggregate a_j.  Its weights are
bf16 values by construction (the caller passes them); the raw inputs x and the
edge features stay float32.  `forward(..., bf16=True)` evaluates it; the
`dtype` argument chooses the accumulation precision (float64 by default;
float32 gives a second, equally valid evaluation of the bf16 model, used to
measure how far rounding-order differences alone move its logits).

Every routine works on plain numpy arrays; the matrix product, argsort and
np.add.at are the only library primitives used.
"""
from __future__ import annotations

import numpy as np

MLP_NAMES = ("node_encoder", "edge_encoder", "edge_network", "node_network", "edge_classifier")


def layer_norm(v: np.ndarray, gamma: np.ndarray, beta: np.ndarray, eps: float) -> np.ndarray:
    """LayerNorm over the last axis with biased variance and affine gamma, beta."""
    mu = v.mean(axis=-1, keepdims=True)
    var = ((v - mu) ** 2).mean(axis=-1, keepdims=True)
    return gamma * (v - mu) / np.sqrt(var + eps) + beta


def relu(v: np.ndarray) -> np.ndarray:
    return np.maximum(v, 0.0)


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Nearest bfloat16 value (8 significant bits, ties to even) of each element, as float64.

    Written from the format's definition: a = m * 2^e with 0.5 <= |m| < 1; the
    nearest value with 8 significant bits is rint(m * 2^8) * 2^(e - 8), where
    rint rounds halfway cases to even.  (Magnitudes here stay far from the
    bfloat16 overflow and subnormal ranges.)"""
    a = np.asarray(a, dtype=np.float64)
    m, e = np.frexp(a)
    return np.ldexp(np.rint(m * 256.0), e - 8)


def mlp(v: np.ndarray, layers, eps: float, act=None, dtype=np.float64) -> np.ndarray:
    """Stack of Linear -> LayerNorm -> ReLU layers; `layers` = [(W [out,in], b, gamma, beta)].
    `act`, when given, is applied to every layer's output (the bf16 model rounds there)."""
    v = np.asarray(v, dtype=dtype)
    for (W, b, g, be) in layers:
        W = np.asarray(W, dtype)
        v = relu(layer_norm(v @ W.T + np.asarray(b, dtype),
                            np.asarray(g, dtype), np.asarray(be, dtype), dtype(eps)))
        if act is not None:
            v = act(v).astype(dtype)
    return v


def wrap_dphi_f32(d: np.ndarray) -> np.ndarray:
    """Wrap float32 phi differences (units of pi) into (-1, 1], in float32."""
    d = np.asarray(d, dtype=np.float32)
    two = np.float32(2.0)
    out = np.where(d > np.float32(1.0), d - two, d)
    out = np.where(out <= np.float32(-1.0), out + two, out)
    return out.astype(np.float32)


def edge_features(x: np.ndarray, src: np.ndarray, dst: np.ndarray) -> np.ndarray:
    """f_ij = (dr, dphi) for every edge i -> j, computed in float32 (see module doc)."""
    x = np.asarray(x, dtype=np.float32)
    dr = (x[dst, 0] - x[src, 0]).astype(np.float32)
    dphi = wrap_dphi_f32((x[dst, 1] - x[src, 1]).astype(np.float32))
    return np.stack([dr, dphi], axis=1)


def csr_by_destination(src: np.ndarray, dst: np.ndarray, n_nodes: int):
    """Destination-keyed CSR: edges stably sorted by destination (ties keep input
    order).  Returns rowptr [N+1], src_sorted [E], perm [E] (sorted slot -> input id)."""
    dst = np.asarray(dst, dtype=np.int64)
    perm = np.argsort(dst, kind="stable")
    counts = np.bincount(dst, minlength=n_nodes) if dst.size else np.zeros(n_nodes, np.int64)
    rowptr = np.zeros(n_nodes + 1, dtype=np.int64)
    rowptr[1:] = np.cumsum(counts)
    return rowptr, np.asarray(src, np.int64)[perm], perm


def aggregate(m: np.ndarray, dst: np.ndarray, n_nodes: int, dtype=np.float64) -> np.ndarray:
    """a_j = sum of the messages of all edges whose destination is j (0 if none)."""
    a = np.zeros((n_nodes, m.shape[1]), dtype=dtype)
    np.add.at(a, np.asarray(dst, np.int64), m)
    return a


def sigmoid(z: np.ndarray) -> np.ndarray:
    z = np.asarray(z, dtype=np.float64)
    return np.where(z >= 0, 1.0 / (1.0 + np.exp(-np.abs(z))),
                    np.exp(-np.abs(z)) / (1.0 + np.exp(-np.abs(z))))


def forward(weights: dict, x: np.ndarray, edge_index: np.ndarray, n_iters: int,
            eps: float = 1e-5, return_logits: bool = False, return_states: bool = False,
            bf16: bool = False, dtype=np.float64):
    """Edge scores (input edge order) of the interaction network on one hit graph.

    `weights` maps each MLP name to its [(W, b, gamma, beta)] layers, plus
    'head_w' [H] and 'head_b' [1].  `edge_index` is [2, E] (row 0 source, row 1
    destination).  `bf16` evaluates the bf16 model (activations rounded to
    bfloat16, see the module doc); `dtype` is the accumulation precision.
    Returns scores (and logits / final states on request)."""
    x = np.asarray(x, dtype=np.float32)
    src = np.asarray(edge_index[0], dtype=np.int64)
    dst = np.asarray(edge_index[1], dtype=np.int64)
    n_nodes = x.shape[0]
    act = round_bf16 if bf16 else None
    keep = (lambda v: round_bf16(v).astype(dtype)) if bf16 else (lambda v: v)
    f = edge_features(x, src, dst).astype(dtype)
    h = mlp(x.astype(dtype), weights["node_encoder"], eps, act, dtype)
    e = mlp(f, weights["edge_encoder"], eps, act, dtype)
    for _ in range(n_iters):
        m = mlp(np.concatenate([h[src], h[dst], e], axis=1), weights["edge_network"], eps, act, dtype)
        e = m
        a = keep(aggregate(m, dst, n_nodes, dtype))
        h = mlp(np.concatenate([h, a], axis=1), weights["node_network"], eps, act, dtype)
    c = mlp(np.concatenate([h[src], h[dst], e], axis=1), weights["edge_classifier"], eps, act, dtype)
    logits = (c @ np.asarray(weights["head_w"], dtype) + dtype(np.asarray(weights["head_b"])[0])).astype(np.float64)
    scores = sigmoid(logits)
    out = [scores]
    if return_logits:
        out.append(logits)
    if return_states:
        out.append({"h": h, "e": e})
    return out[0] if len(out) == 1 else tuple(out)


def track_labels(scores: np.ndarray, edge_index: np.ndarray, n_nodes: int, threshold: float = 0.5) -> np.ndarray:
    """Track candidates (Section 2.1: the edge scores are thresholded and the weakly connected
    components of the kept edges are the tracks; Section 2.3: one integer label per space point).

    An edge is kept when its score is > threshold (NaN is never kept) and both endpoints lie in
    [0, n_nodes).  Each hit is labelled by the smallest node id of its component, found by
    repeating  label[u] = label[v] = min(label[u], label[v])  over the kept edges until no label
    changes (labels only decrease, and the smallest id of a component reaches every member)."""
    s = np.asarray(scores, dtype=np.float64)
    u = np.asarray(edge_index[0], dtype=np.int64)
    v = np.asarray(edge_index[1], dtype=np.int64)
    keep = (s > threshold) & (u >= 0) & (u < n_nodes) & (v >= 0) & (v < n_nodes)
    u, v = u[keep], v[keep]
    label = np.arange(n_nodes, dtype=np.int64)
    while True:
        m = np.minimum(label[u], label[v])
        new = label.copy()
        np.minimum.at(new, u, m)
        np.minimum.at(new, v, m)
        if np.array_equal(new, label):
            return label.astype(np.int32)
        label = new


def filter_scores(fw: dict, x: np.ndarray, edge_index: np.ndarray, eps: float = 1e-5, bf16: bool = False,
                  return_logits: bool = False):
    """Filtering step (Section 2.1: before the GNN, an MLP scores every candidate edge from the raw
    features of its two hits): s = sigmoid(w_o . MLP([x_src, x_dst]) + b_o).  `fw` holds 'layers'
    [(W, b, gamma, beta)], 'head_w' [H], 'head_b' [1].  Edges with an endpoint outside
    [0, N) score NaN.  `bf16` rounds every layer output to bfloat16, as in forward()."""
    x = np.asarray(x, dtype=np.float32)
    src = np.asarray(edge_index[0], dtype=np.int64)
    dst = np.asarray(edge_index[1], dtype=np.int64)
    n = x.shape[0]
    ok = (src >= 0) & (src < n) & (dst >= 0) & (dst < n)
    s_, d_ = np.where(ok, src, 0), np.where(ok, dst, 0)
    v = np.concatenate([x[s_], x[d_]], axis=1).astype(np.float64)
    c = mlp(v, fw["layers"], eps, round_bf16 if bf16 else None)
    logits = c @ np.asarray(fw["head_w"], np.float64) + float(np.asarray(fw["head_b"])[0])
    logits = np.where(ok, logits, np.nan)
    scores = sigmoid(np.where(ok, logits, 0.0))
    scores = np.where(ok, scores, np.nan)
    return (scores, logits) if return_logits else scores


def apply_filtering(scores: np.ndarray, edge_index: np.ndarray, threshold: float):
    """applyFiltering (Section 2.1): the edges whose score is > threshold (NaN never), in input
    order.  Returns (kept edge index [2, n_kept], input ids of the kept edges)."""
    keep = np.asarray(scores) > threshold
    ids = np.nonzero(keep)[0]
    return np.asarray(edge_index)[:, ids], ids


def embed(ew: dict, x: np.ndarray, eps: float = 1e-5, bf16: bool = False) -> np.ndarray:
    """Embedding step (Section 2.1: an MLP maps every space point's raw features into a latent
    space): y = normalize(W_out . MLP(x) + b_out), unit length (a zero vector stays zero)."""
    v = mlp(np.asarray(x, np.float64), ew["layers"], eps, round_bf16 if bf16 else None)
    z = v @ np.asarray(ew["out_w"], np.float64).T + np.asarray(ew["out_b"], np.float64)
    n = np.sqrt((z * z).sum(axis=1, keepdims=True))
    return np.where(n > 0, z / np.where(n > 0, n, 1.0), 0.0)


def sq_dist_f32(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """Squared distances of float32 row pairs, summed over the coordinates in order with one
    float32 rounding per product and per sum."""
    a = np.asarray(a, np.float32)
    b = np.asarray(b, np.float32)
    s = np.zeros(a.shape[0], np.float32)
    for d in range(a.shape[1]):
        diff = (a[:, d] - b[:, d]).astype(np.float32)
        s = (s + (diff * diff).astype(np.float32)).astype(np.float32)
    return s


def radius_graph(emb: np.ndarray, r_col: np.ndarray, radius: float, candidates=None) -> np.ndarray:
    """Graph building (Section 2.1: edges between hits closer than a radius in the latent space):
    every pair {i, j} whose float32 squared distance (sq_dist_f32) is below float32(radius)^2
    (rounded to float32), oriented from the smaller r (r_col; the smaller index on a tie) to the
    other.  Returns the edges as an [n, 2] array sorted by (src, dst).  `candidates` ([m, 2], i < j)
    may restrict the pairs tested (a superset of the answer); by default every pair is tested."""
    emb = np.asarray(emb, np.float32)
    n = emb.shape[0]
    if candidates is None:
        ii, jj = np.triu_indices(n, 1)
    else:
        ii, jj = candidates[:, 0], candidates[:, 1]
    r2 = np.float32(np.float32(radius) * np.float32(radius))
    keep = sq_dist_f32(emb[ii], emb[jj]) < r2
    i, j = ii[keep], jj[keep]
    r = np.asarray(r_col, np.float32)
    first = (r[i] < r[j]) | ((r[i] == r[j]) & (i < j))
    e = np.stack([np.where(first, i, j), np.where(first, j, i)], axis=1).astype(np.int64)
    return e[np.lexsort((e[:, 1], e[:, 0]))] if e.size else e.reshape(0, 2)

