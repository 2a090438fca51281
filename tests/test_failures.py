"""Failure detection without a GPU fault.

CPU: malformed weight blobs are rejected before any device work.  GPU (marked): allocation failures
injected on the host return GNN_ERR_OOM and leave the context usable; a bounded device wait that
expires (an mbarrier nothing completes) is reported by gnn_status as GNN_ERR_DEVICE_TIMEOUT, after
which the context still scores correctly."""
import ctypes
import struct

import numpy as np
import pytest

from paper_2402_09633_gb300 import synthetic as S

CFG = S.ModelConfig(3, 2, 64, 2, 2)


def _lib():
    from paper_2402_09633_gb300 import binding
    lib = binding.load_library()
    lib.gnn_debug_fail_allocs.argtypes = [ctypes.c_int]
    lib.gnn_debug_fail_allocs.restype = ctypes.c_int
    lib.gnn_debug_wait_timeout.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]
    lib.gnn_debug_wait_timeout.restype = ctypes.c_int
    return lib


def _create(blob, cfg=CFG):
    from paper_2402_09633_gb300 import binding
    lib = binding.load_library()
    c = binding.GnnConfig(1, cfg.n_node_feat, cfg.n_edge_feat, cfg.hidden, cfg.n_iters, cfg.mlp_layers,
                          cfg.precision, cfg.ln_eps)
    h = ctypes.c_void_p()
    buf = ctypes.create_string_buffer(blob, len(blob))
    rc = lib.gnn_create(ctypes.byref(c), buf, len(blob), ctypes.byref(h))
    if rc == 0:
        lib.gnn_destroy(h)
    return rc


def test_malformed_blobs_rejected_before_device_work():
    blob = S.pack_blob(CFG, S.init_weights(CFG, 0))
    bad_magic = b"XXXX" + blob[4:]
    assert _create(bad_magic) == -2
    assert _create(blob[:-4]) == -2                            # truncated payload
    assert _create(blob + b"\0\0\0\0") == -2                   # trailing bytes
    assert _create(blob[:20]) == -2                            # shorter than the header
    other = S.ModelConfig(3, 2, 64, 3, 2)                     # header says T=2, config T=3
    assert _create(blob, other) == -2
    hdr = list(struct.unpack("<8i", blob[:32]))
    hdr[1] = 2                                                 # unknown blob version
    assert _create(struct.pack("<8i", *hdr) + blob[32:]) == -2


def test_fail_allocs_argument_check():
    assert _lib().gnn_debug_fail_allocs(-1) == -1
    assert _lib().gnn_debug_fail_allocs(0) == 0


@pytest.mark.gpu
def test_injected_allocation_failures_leave_context_usable():
    import torch
    from paper_2402_09633_gb300 import GnnError, InteractionNetwork
    from tests.gpu_util import check_parity
    lib = _lib()
    W = S.init_weights(CFG, 0)
    blob = S.pack_blob(CFG, W)
    lib.gnn_debug_fail_allocs(1)
    with pytest.raises(GnnError) as ex:
        InteractionNetwork(CFG, blob)
    assert ex.value.code == -3
    net = InteractionNetwork(CFG, blob)                       # the failure was consumed
    x, ei = S.random_graph(500, 2000, 3, 1)
    xs, es = torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda()
    lib.gnn_debug_fail_allocs(1)
    with pytest.raises(GnnError) as ex:                       # workspace growth fails
        net.infer(xs, es)
    assert ex.value.code == -3
    lib.gnn_debug_fail_allocs(1)
    with pytest.raises(GnnError) as ex:
        net.reserve(1000, 5000)
    assert ex.value.code == -3
    s = net.infer(xs, es).cpu().numpy()                       # and then works
    assert net.status() == 0
    check_parity(s, W, x, ei, CFG.n_iters)
    host = np.empty(ei.shape[1], np.float32)
    lib.gnn_debug_fail_allocs(1)
    with pytest.raises(GnnError) as ex:                       # staging of the host entry point
        net.infer_host(x, ei, host)
    assert ex.value.code == -3
    assert net.infer_host(x, ei, host) == 0 and host.tobytes() == s.tobytes()
    net.close()


@pytest.mark.gpu
def test_expired_device_wait_is_reported_and_context_stays_usable():
    import torch
    from paper_2402_09633_gb300 import InteractionNetwork
    from tests.gpu_util import check_parity
    lib = _lib()
    W = S.init_weights(CFG, 2)
    net = InteractionNetwork(CFG, S.pack_blob(CFG, W))
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert lib.gnn_debug_wait_timeout(net.handle, 0, stream) == -1
    assert lib.gnn_debug_wait_timeout(net.handle, 50_000_000, stream) == 0     # 50 ms
    assert net.status() == -6                                  # DEVICE_TIMEOUT, then cleared
    assert net.status() == 0
    x, ei = S.random_graph(300, 1200, 3, 3)
    s = net.infer(torch.from_numpy(x).cuda(), torch.from_numpy(ei).cuda()).cpu().numpy()
    assert net.status() == 0
    check_parity(s, W, x, ei, CFG.n_iters)
    net.close()
