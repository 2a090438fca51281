"""Seeded synthetic inputs for the interaction-network edge classifier.

This module draws the random numbers both sides of every parity check use:
hit graphs shaped like the paper's events (about 300k space points and 1M
candidate edges per event, Section 1; space points on concentric detector
layers, candidate edges between neighbouring layers, Section 2.1) and the
random-init weights of the network, packed into the weight blob that
``gnn_create`` parses.  It holds none of the method's arithmetic: no layer,
normalisation, aggregation or score is computed here.

Node features (columns): 0 = r/1000, 1 = phi/pi, 2 = z/1000, then optional
extra features ~ N(0, 1) (the cluster-shape stand-ins of the 12-feature
workloads).  Edge index: int32 [2, E], row 0 = source (inner layer), row 1 =
destination (outer layer), in a seeded shuffled order.
"""
from __future__ import annotations

import struct
from dataclasses import dataclass, field

import numpy as np

# Detector layer radii in mm (10 concentric cylinders).
LAYER_RADII_MM = (32.0, 72.0, 116.0, 172.0, 260.0, 360.0, 500.0, 600.0, 700.0, 820.0)
N_LAYERS = len(LAYER_RADII_MM)
MAX_IN_DEGREE = 40

BLOB_MAGIC = 0x57474E47  # "GNGW" little-endian
BLOB_VERSION = 1
# Order of the five MLPs inside the blob.
MLP_NAMES = ("node_encoder", "edge_encoder", "edge_network", "node_network", "edge_classifier")

PRECISION_FP32 = 0   # fp32 storage, split-bf16 (three-product) tensor-core math
PRECISION_BF16 = 1   # bf16 weights and stored state, fp32 accumulate


@dataclass(frozen=True)
class ModelConfig:
    n_node_feat: int = 3
    n_edge_feat: int = 2
    hidden: int = 128
    n_iters: int = 8
    mlp_layers: int = 3
    precision: int = PRECISION_FP32
    ln_eps: float = 1e-5

    def mlp_in_dims(self):
        H = self.hidden
        return {"node_encoder": self.n_node_feat, "edge_encoder": self.n_edge_feat,
                "edge_network": 3 * H, "node_network": 2 * H, "edge_classifier": 3 * H}


@dataclass(frozen=True)
class EventSpec:
    """Shape of one synthetic event."""
    n_nodes: int
    n_extra_feat: int = 0          # extra N(0,1) node features beyond (r, phi, z)
    mode: str = "fanout"           # "fanout": each inner node links to <=4 next-layer nodes
                                   # "powerlaw": power-law in-degree, exact edge count
    dphi_window: float = 0.3       # |dphi| window in radians
    fanout: int = 4
    n_edges: int = 0               # "powerlaw" only: exact total


@dataclass(frozen=True)
class Workload:
    name: str
    model: ModelConfig
    event: EventSpec
    n_events: int = 1
    seeds: tuple = (0,)
    weight_seed: int = 0
    description: str = ""


# The five workloads of the edge-classification benchmark.
WORKLOADS = {
    "tiny": Workload("tiny", ModelConfig(3, 2, 64, 4, 2), EventSpec(2000, 0, "fanout", 0.3),
                     description="2,000 nodes / ~7.2k edges, fp32, H=64, T=4, 2-layer MLPs"),
    "mid": Workload("mid", ModelConfig(3, 2, 128, 8, 3), EventSpec(30000, 0, "fanout", 0.1),
                    description="30,000 nodes / ~108k edges, fp32, H=128, T=8, 3-layer MLPs"),
    "full": Workload("full", ModelConfig(12, 2, 128, 8, 3),
                     EventSpec(300000, 9, "powerlaw", 0.02, n_edges=1_000_000),
                     description="300,000 nodes / 1,000,000 edges, 12 features, fp32 model, H=128, T=8"),
    "full_bf16": Workload("full_bf16", ModelConfig(12, 2, 128, 8, 3, PRECISION_BF16),
                          EventSpec(300000, 9, "powerlaw", 0.02, n_edges=1_000_000),
                          description="as 'full' with bf16 weights and stored state"),
    "batch16": Workload("batch16", ModelConfig(12, 2, 128, 8, 3),
                        EventSpec(300000, 9, "powerlaw", 0.02, n_edges=1_000_000),
                        n_events=16, seeds=tuple(range(16)),
                        description="16 full events as one block-diagonal graph (4.8M nodes, 16M edges)"),
}


def _layer_of(n_nodes: int) -> np.ndarray:
    """Layer id of every node: equal counts per layer (remainder on the last layers)."""
    base = n_nodes // N_LAYERS
    counts = np.full(N_LAYERS, base, dtype=np.int64)
    counts[N_LAYERS - (n_nodes - base * N_LAYERS):] += 1 if n_nodes % N_LAYERS else 0
    return np.repeat(np.arange(N_LAYERS), counts)


def _powerlaw_alpha(mean: float, dmax: int = MAX_IN_DEGREE) -> float:
    """Exponent a of p(d) ~ (d+1)^-a on {0..dmax} whose mean is `mean` (bisection)."""
    d = np.arange(dmax + 1, dtype=np.float64)
    lo, hi = 0.0, 10.0
    for _ in range(200):
        a = 0.5 * (lo + hi)
        p = (d + 1.0) ** -a
        m = (d * p).sum() / p.sum()
        if m > mean:
            lo = a
        else:
            hi = a
    return 0.5 * (lo + hi)


def _window(sorted_phi: np.ndarray, phi_q: np.ndarray, half: float, need: np.ndarray):
    """Index window [lo, hi) into the 3x-extended (wrapped) sorted phi array holding
    every candidate within |dphi| < half of each query, widened to >= need entries."""
    n = sorted_phi.size
    ext = np.concatenate([sorted_phi - 2 * np.pi, sorted_phi, sorted_phi + 2 * np.pi])
    lo = np.searchsorted(ext, phi_q - half, side="right")
    hi = np.searchsorted(ext, phi_q + half, side="left")
    short = (hi - lo) < need
    if np.any(short):
        c = np.searchsorted(ext, phi_q[short])
        w = need[short]
        lo[short] = c - (w + 1) // 2
        hi[short] = lo[short] + w
    width = np.minimum(hi - lo, n)
    return lo, lo + width


def _distinct_picks(rng, width: np.ndarray, count: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """For each query q, `count[q]` distinct offsets in [0, width[q]) (uniform)."""
    owner = np.repeat(np.arange(width.size), count)
    pos = np.floor(rng.random(owner.size) * width[owner]).astype(np.int64)
    while True:
        key = owner * (int(width.max()) + 1) + pos
        order = np.argsort(key, kind="stable")
        dup = np.zeros(owner.size, dtype=bool)
        dup[order[1:]] = key[order[1:]] == key[order[:-1]]
        if not dup.any():
            return owner, pos
        pos[dup] = np.floor(rng.random(int(dup.sum())) * width[owner[dup]]).astype(np.int64)


def generate_event(spec: EventSpec, seed: int = 0):
    """One synthetic event: (x float32 [N, 3+extra], edge_index int32 [2, E])."""
    rng = np.random.default_rng(seed)
    N = spec.n_nodes
    layer = _layer_of(N)
    r = np.asarray(LAYER_RADII_MM)[layer]
    phi = rng.uniform(-np.pi, np.pi, N)
    z = rng.uniform(-1000.0, 1000.0, N)
    cols = [r / 1000.0, phi / np.pi, z / 1000.0]
    if spec.n_extra_feat:
        cols += list(rng.standard_normal((spec.n_extra_feat, N)))
    x = np.stack(cols, axis=1).astype(np.float32)
    phi = x[:, 1].astype(np.float64) * np.pi      # the stored (fp32) phi decides the windows

    starts = np.searchsorted(layer, np.arange(N_LAYERS + 1))
    srcs, dsts = [], []
    if spec.mode == "fanout":
        for l in range(N_LAYERS - 1):
            a0, a1, b0, b1 = starts[l], starts[l + 1], starts[l + 1], starts[l + 2]
            order = b0 + np.argsort(phi[b0:b1], kind="stable")
            sp = phi[order]
            q = np.arange(a0, a1)
            lo, hi = _window(sp, phi[q], spec.dphi_window, np.zeros(q.size, np.int64))
            # keep only true in-window candidates (no widening in this mode)
            width = hi - lo
            count = np.minimum(spec.fanout, width)
            owner, pos = _distinct_picks(rng, np.maximum(width, 1), count)
            tgt = order[(lo[owner] + pos) % sp.size]
            srcs.append(q[owner]); dsts.append(tgt)
    elif spec.mode == "powerlaw":
        inner = starts[1]                 # nodes on layers 1..9 receive edges
        n_recv = N - inner
        alpha = _powerlaw_alpha(spec.n_edges / n_recv)
        dvals = np.arange(MAX_IN_DEGREE + 1)
        p = (dvals + 1.0) ** -alpha
        deg = rng.choice(dvals, size=n_recv, p=p / p.sum())
        diff = spec.n_edges - int(deg.sum())
        order = rng.permutation(n_recv)
        while diff != 0:                  # deterministic fix-up to the exact total
            step = 1 if diff > 0 else -1
            ok = order[(deg[order] < MAX_IN_DEGREE) if step > 0 else (deg[order] > 0)]
            take = ok[:abs(diff)]
            deg[take] += step
            diff -= step * take.size
        deg_full = np.zeros(N, np.int64)
        deg_full[inner:] = deg
        for l in range(1, N_LAYERS):
            a0, a1, b0, b1 = starts[l - 1], starts[l], starts[l], starts[l + 1]
            order_s = a0 + np.argsort(phi[a0:a1], kind="stable")
            sp = phi[order_s]
            q = np.arange(b0, b1)
            need = np.minimum(deg_full[q], sp.size)
            lo, hi = _window(sp, phi[q], spec.dphi_window, need)
            owner, pos = _distinct_picks(rng, hi - lo, need)
            srcs.append(order_s[(lo[owner] + pos) % sp.size]); dsts.append(q[owner])
    else:
        raise ValueError(spec.mode)
    src = np.concatenate(srcs).astype(np.int64)
    dst = np.concatenate(dsts).astype(np.int64)
    shuffle = rng.permutation(src.size)
    edge_index = np.stack([src[shuffle], dst[shuffle]]).astype(np.int32)
    return x, edge_index


def generate_batch(spec: EventSpec, seeds) -> tuple[np.ndarray, np.ndarray]:
    """Independent events concatenated block-diagonally (node ids offset per event)."""
    xs, eis, off = [], [], 0
    for s in seeds:
        x, ei = generate_event(spec, s)
        xs.append(x); eis.append(ei.astype(np.int64) + off); off += x.shape[0]
    return np.concatenate(xs), np.concatenate(eis, axis=1).astype(np.int32)


def random_graph(n_nodes: int, n_edges: int, n_feat: int, seed: int = 0):
    """Unstructured graph for edge cases: uniform endpoints (duplicates and
    self-loops allowed), node features ~ N(0,1) with column 1 in [-1, 1)."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((n_nodes, n_feat)).astype(np.float32)
    if n_feat > 1:
        x[:, 1] = rng.uniform(-1.0, 1.0, n_nodes).astype(np.float32)
    ei = rng.integers(0, max(n_nodes, 1), size=(2, n_edges)).astype(np.int32)
    return x, ei


# --------------------------------------------------------------------------- weights

def _round_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even), kept as float32."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def init_weights(cfg: ModelConfig, seed: int = 0) -> dict:
    """Random-init weights: W ~ N(0, 1/fan_in), b ~ N(0, 0.1^2), gamma = 1 + N(0, 0.1^2),
    beta ~ N(0, 0.1^2); head w_o ~ N(0, 1/H), b_o = 0.  Draws follow blob order.
    For the bf16 model every value is rounded to bf16 (the model's weights are bf16)."""
    rng = np.random.default_rng(seed)
    H = cfg.hidden
    dims = cfg.mlp_in_dims()
    out = {}
    for name in MLP_NAMES:
        layers = []
        fan_in = dims[name]
        for l in range(cfg.mlp_layers):
            W = (rng.standard_normal((H, fan_in)) / np.sqrt(fan_in)).astype(np.float32)
            b = (0.1 * rng.standard_normal(H)).astype(np.float32)
            g = (1.0 + 0.1 * rng.standard_normal(H)).astype(np.float32)
            be = (0.1 * rng.standard_normal(H)).astype(np.float32)
            layers.append((W, b, g, be))
            fan_in = H
        out[name] = layers
    out["head_w"] = (rng.standard_normal(H) / np.sqrt(H)).astype(np.float32)
    out["head_b"] = np.zeros(1, np.float32)
    if cfg.precision == PRECISION_BF16:
        out = {k: ([tuple(_round_bf16(t) for t in lay) for lay in v] if isinstance(v, list)
                   else _round_bf16(v)) for k, v in out.items()}
    return out


def pack_blob(cfg: ModelConfig, weights: dict) -> bytes:
    """Flat little-endian blob: header of 8 int32 + 1 float32 + 1 int64 count, then
    float32 arrays: per MLP (blob order), per layer: W [H, in] row-major, b, gamma,
    beta; then head_w [H], head_b [1]."""
    arrays = []
    for name in MLP_NAMES:
        for (W, b, g, be) in weights[name]:
            arrays += [W, b, g, be]
    arrays += [weights["head_w"], weights["head_b"]]
    payload = b"".join(np.ascontiguousarray(a, dtype="<f4").tobytes() for a in arrays)
    n_floats = len(payload) // 4
    header = struct.pack("<8i f i q", BLOB_MAGIC, BLOB_VERSION, cfg.n_node_feat, cfg.n_edge_feat,
                         cfg.hidden, cfg.n_iters, cfg.mlp_layers, cfg.precision, cfg.ln_eps,
                         0, n_floats)
    return header + payload


BLOB_HEADER_BYTES = struct.calcsize("<8i f i q")


def blob_n_floats(cfg: ModelConfig) -> int:
    H, L = cfg.hidden, cfg.mlp_layers
    n = 0
    for name, fan_in in cfg.mlp_in_dims().items():
        n += H * fan_in + 3 * H + (L - 1) * (H * H + 3 * H)
    return n + H + 1


# --------------------------------------------------------------------------- filtering MLP

FILTER_MAGIC = 0x4C464E47  # "GNFL" little-endian


def init_filter_weights(cfg: ModelConfig, seed: int = 1) -> dict:
    """Random-init filtering MLP on [x_src, x_dst] (2 * n_node_feat inputs): layers of the same
    kind and draws as init_weights, then head w_o ~ N(0, 1/H), b_o = 0; rounded to bf16 for the
    bf16 model."""
    rng = np.random.default_rng(seed)
    H = cfg.hidden
    fan_in = 2 * cfg.n_node_feat
    layers = []
    for _ in range(cfg.mlp_layers):
        W = (rng.standard_normal((H, fan_in)) / np.sqrt(fan_in)).astype(np.float32)
        b = (0.1 * rng.standard_normal(H)).astype(np.float32)
        g = (1.0 + 0.1 * rng.standard_normal(H)).astype(np.float32)
        be = (0.1 * rng.standard_normal(H)).astype(np.float32)
        layers.append((W, b, g, be))
        fan_in = H
    out = {"layers": layers, "head_w": (rng.standard_normal(H) / np.sqrt(H)).astype(np.float32),
           "head_b": np.zeros(1, np.float32)}
    if cfg.precision == PRECISION_BF16:
        out = {"layers": [tuple(_round_bf16(t) for t in lay) for lay in layers],
               "head_w": _round_bf16(out["head_w"]), "head_b": _round_bf16(out["head_b"])}
    return out


def pack_filter_blob(cfg: ModelConfig, fw: dict) -> bytes:
    """Filter blob: 8 int32 (magic, version 1, n_node_feat, hidden, mlp_layers, precision, 0, 0),
    float32 ln_eps, int32 0, int64 float count; per layer W [H, in], b, gamma, beta; w_o, b_o."""
    arrays = []
    for (W, b, g, be) in fw["layers"]:
        arrays += [W, b, g, be]
    arrays += [fw["head_w"], fw["head_b"]]
    payload = b"".join(np.ascontiguousarray(a, dtype="<f4").tobytes() for a in arrays)
    header = struct.pack("<8i f i q", FILTER_MAGIC, 1, cfg.n_node_feat, cfg.hidden, len(fw["layers"]),
                         cfg.precision, 0, 0, cfg.ln_eps, 0, len(payload) // 4)
    return header + payload


# --------------------------------------------------------------------------- embedding MLP

EMBED_MAGIC = 0x4D454E47  # "GNEM" little-endian


def init_embed_weights(cfg: ModelConfig, dim: int = 8, seed: int = 2) -> dict:
    """Random-init embedding MLP: mlp_layers hidden layers on x (n_node_feat inputs) drawn as in
    init_weights, then W_out [dim, H] ~ N(0, 1/H) and b_out ~ N(0, 0.1^2); bf16-rounded for the
    bf16 model."""
    rng = np.random.default_rng(seed)
    H = cfg.hidden
    fan_in = cfg.n_node_feat
    layers = []
    for _ in range(cfg.mlp_layers):
        W = (rng.standard_normal((H, fan_in)) / np.sqrt(fan_in)).astype(np.float32)
        b = (0.1 * rng.standard_normal(H)).astype(np.float32)
        g = (1.0 + 0.1 * rng.standard_normal(H)).astype(np.float32)
        be = (0.1 * rng.standard_normal(H)).astype(np.float32)
        layers.append((W, b, g, be))
        fan_in = H
    out = {"layers": layers, "out_w": (rng.standard_normal((dim, H)) / np.sqrt(H)).astype(np.float32),
           "out_b": (0.1 * rng.standard_normal(dim)).astype(np.float32)}
    if cfg.precision == PRECISION_BF16:
        out = {"layers": [tuple(_round_bf16(t) for t in lay) for lay in layers],
               "out_w": _round_bf16(out["out_w"]), "out_b": _round_bf16(out["out_b"])}
    return out


def pack_embed_blob(cfg: ModelConfig, ew: dict) -> bytes:
    """Embedding blob: 8 int32 (magic, version 1, n_node_feat, hidden, layers, precision, dim, 0),
    float32 ln_eps, int32 0, int64 float count; per layer W, b, gamma, beta; W_out [dim, H], b_out."""
    arrays = []
    for (W, b, g, be) in ew["layers"]:
        arrays += [W, b, g, be]
    arrays += [ew["out_w"], ew["out_b"]]
    payload = b"".join(np.ascontiguousarray(a, dtype="<f4").tobytes() for a in arrays)
    header = struct.pack("<8i f i q", EMBED_MAGIC, 1, cfg.n_node_feat, cfg.hidden, len(ew["layers"]),
                         cfg.precision, ew["out_w"].shape[0], 0, cfg.ln_eps, 0, len(payload) // 4)
    return header + payload

