"""The allocation-free CSR entry point (gnn_csr_build_noalloc) against gnn_infer's own CSR.

Some callers may not allocate device memory once they are running (a serving
process whose memory planner owns every allocation, or request paths that
must not pay cudaMalloc's implicit synchronisation).  gnn_csr_build_noalloc
serves them from a fixed library-owned scratch array.  This test calls it
through the C ABI twice in a row, a large graph and then a smaller one (so
stale scratch contents from the first call would show), and requires
bit-identical CSR arrays to the ones gnn_infer builds for the same edges.
This file is collected last on purpose."""
import ctypes

import numpy as np
import pytest

from oracle import gnn_oracle as O
from paper_2402_09633_gb300 import synthetic as S

pytestmark = pytest.mark.gpu

MAX_EDGES = 1 << 20


def _lib():
    from paper_2402_09633_gb300 import binding
    lib = binding.load_library()
    vp, i64 = ctypes.c_void_p, ctypes.c_int64
    lib.gnn_csr_build_noalloc.argtypes = [vp, i64, i64, vp, vp, vp, vp]
    lib.gnn_csr_build_noalloc.restype = ctypes.c_int
    return lib


def _noalloc_csr(lib, ei_dev, n, e):
    import torch
    rowptr = torch.full((n + 1,), -7, dtype=torch.int32, device="cuda")
    perm = torch.full((max(e, 1),), -7, dtype=torch.int32, device="cuda")
    src = torch.full((max(e, 1),), -7, dtype=torch.int32, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = lib.gnn_csr_build_noalloc(ctypes.c_void_p(ei_dev.data_ptr()), n, e, ctypes.c_void_p(rowptr.data_ptr()),
                                   ctypes.c_void_p(perm.data_ptr()), ctypes.c_void_p(src.data_ptr()), stream)
    torch.cuda.synchronize()
    return rc, rowptr.cpu().numpy(), perm.cpu().numpy()[:e], src.cpu().numpy()[:e]


def _infer_csr(x, ei):
    """The CSR gnn_infer builds (read back through gnn_debug_copy)."""
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    cfg = S.ModelConfig(x.shape[1], 2, 64, 1, 2)
    net = InteractionNetwork(cfg, S.pack_blob(cfg, S.init_weights(cfg, 0)))
    net.infer(torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda())
    n, e = x.shape[0], ei.shape[1]
    out = (net.debug_copy(0, (n + 1,), torch.int32).cpu().numpy(),
           net.debug_copy(1, (e,), torch.int32).cpu().numpy(),
           net.debug_copy(2, (e,), torch.int32).cpu().numpy())
    net.close()
    return out


def test_noalloc_csr_matches_gnn_infer_on_two_calls_in_a_row():
    import torch
    lib = _lib()
    big = S.generate_event(S.EventSpec(300000, 9, "powerlaw", 0.02, n_edges=MAX_EDGES), 3)
    small = S.random_graph(777, 5001, 3, seed=4)            # duplicates and self-loops included
    for x, ei in (big, small):
        n, e = x.shape[0], ei.shape[1]
        rc, rowptr, perm, src = _noalloc_csr(lib, torch.from_numpy(ei).cuda(), n, e)
        assert rc == 0
        want_rowptr, want_perm, want_src = _infer_csr(x, ei)
        np.testing.assert_array_equal(rowptr, want_rowptr)
        np.testing.assert_array_equal(perm, want_perm)
        np.testing.assert_array_equal(src, want_src)
        o_rowptr, o_src, o_perm = O.csr_by_destination(ei[0], ei[1], n)
        np.testing.assert_array_equal(perm, o_perm)


def test_noalloc_csr_limits_and_empty_graph():
    import torch
    lib = _lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    dummy = torch.zeros(16, dtype=torch.int32, device="cuda")
    p = ctypes.c_void_p(dummy.data_ptr())
    assert lib.gnn_csr_build_noalloc(p, 10, MAX_EDGES + 1, p, p, p, stream) == -1     # beyond the maximum
    assert lib.gnn_csr_build_noalloc(p, -1, 4, p, p, p, stream) == -1
    assert lib.gnn_csr_build_noalloc(None, 10, 4, p, p, p, stream) == -1
    rc, rowptr, _, _ = _noalloc_csr(lib, dummy, 9, 0)                                  # no edges
    assert rc == 0 and rowptr.tolist() == [0] * 10


def test_noalloc_csr_out_of_range_endpoints():
    """Edges with an endpoint outside [0, n_nodes) sort after rowptr[n_nodes], in input order, with
    source 0; the valid edges form the oracle's CSR of the valid subset.  The call has no error word,
    so rowptr[n_nodes] < n_edges is the caller's only signal, and it must hold here."""
    import torch
    lib = _lib()
    n = 50
    x, ei = S.random_graph(n, 600, 3, seed=9)
    ei = ei.copy()
    rng = np.random.default_rng(5)
    bad = rng.choice(ei.shape[1], 40, replace=False)
    ei[0, bad[:10]] = -1 - rng.integers(0, 5, 10)                  # negative sources
    ei[1, bad[10:20]] = n + rng.integers(0, 7, 10)                 # destinations past the last node
    ei[0, bad[20:30]] = n
    ei[1, bad[30:]] = -3
    e = ei.shape[1]
    rc, rowptr, perm, src = _noalloc_csr(lib, torch.from_numpy(ei).cuda(), n, e)
    assert rc == 0
    valid = (ei[0] >= 0) & (ei[0] < n) & (ei[1] >= 0) & (ei[1] < n)
    ids = np.flatnonzero(valid)
    o_rowptr, o_src, o_perm = O.csr_by_destination(ei[0, ids], ei[1, ids], n)
    assert rowptr[n] == ids.size < e
    np.testing.assert_array_equal(rowptr, o_rowptr)
    np.testing.assert_array_equal(perm[:ids.size], ids[o_perm])
    np.testing.assert_array_equal(src[:ids.size], o_src)
    np.testing.assert_array_equal(perm[ids.size:], np.flatnonzero(~valid))
    np.testing.assert_array_equal(src[ids.size:], 0)
