"""Helpers shared by the GPU parity tests (host-side marshalling and comparisons)."""
import numpy as np

from oracle import gnn_oracle as O
from paper_2402_09633_gb300 import synthetic as S

LOGIT_TOL_FP32 = 2e-3      # max |logit_gpu - logit_oracle| for the fp32 path
DECISION_MARGIN = 1e-2     # decisions must agree where |oracle logit| exceeds this


def logits_from_scores(s):
    s = np.asarray(s, dtype=np.float64)
    return np.log(s) - np.log1p(-s)


def run_gpu(cfg, W, x, ei, reserve=None, return_net=False):
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    net = InteractionNetwork(cfg, S.pack_blob(cfg, W))
    if reserve:
        net.reserve(*reserve)
    xs = torch.from_numpy(np.ascontiguousarray(x)).cuda()
    es = torch.from_numpy(np.ascontiguousarray(ei)).cuda()
    s = net.infer(xs, es)
    rc = net.status()
    out = s.cpu().numpy()
    if return_net:
        return out, rc, net
    net.close()
    return out, rc


def check_parity(s_gpu, W, x, ei, T, tol=LOGIT_TOL_FP32, eps=1e-5):
    _, want = O.forward(W, x, ei, T, eps, return_logits=True)
    assert np.all(np.isfinite(s_gpu)), "non-finite GPU score"
    assert np.all((s_gpu > 0) & (s_gpu < 1)), "saturated score: logit not recoverable"
    got = logits_from_scores(s_gpu)
    err = np.abs(got - want)
    assert err.max() <= tol, f"max logit error {err.max():.3e} at edge {int(err.argmax())}"
    sure = np.abs(want) > DECISION_MARGIN
    assert np.array_equal(got[sure] > 0, want[sure] > 0), "edge decision mismatch"
    return float(err.max())


def untile(buf, n_rows, H):
    """Row-tiled state (T16 layout, see gnn_debug_copy in include/gnn.h) -> row-major [n_rows, H]."""
    R = (n_rows + 127) // 128 * 128
    c = np.arange(H)
    b = c // 8
    x = 4 * ((c % 8) // 2) + 2 * (b % 2) + c % 2
    r = np.arange(R)
    idx = (((r[:, None] // 128) * (H // 16) + (b // 2)[None, :]) * 2048 + (r[:, None] % 128) * 16 + x[None, :])
    return np.asarray(buf)[idx][:n_rows]
