"""ctypes binding of the C ABI in include/gnn.h (argument marshalling only).

Device memory and streams come from PyTorch tensors; every step of the
computation runs in the library's CUDA kernels."""
from __future__ import annotations

import ctypes
import struct
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libgnn_gb300.so")
_lib = None

GNN_OK = 0
ERRORS = {-1: "INVALID_ARG", -2: "BAD_WEIGHTS", -3: "OOM", -4: "CUDA", -5: "INDEX_RANGE",
          -6: "DEVICE_TIMEOUT", -7: "CAPACITY"}
EXPORTED = ("gnn_create", "gnn_reserve", "gnn_infer", "gnn_infer_host", "gnn_status",
            "gnn_destroy", "gnn_error_string", "gnn_debug_copy", "gnn_profile_enable",
            "gnn_profile_read", "gnn_track_labels", "gnn_csr_build_noalloc", "gnn_filter_load",
            "gnn_filter_edges", "gnn_embed_load", "gnn_embed", "gnn_build_graph")
PROFILE_GROUPS = ("csr_build", "node_encoder", "edge_encoder", "edge_update", "node_update",
                  "classifier", "host_copies", "aggregate", "filter", "embed")


class GnnError(RuntimeError):
    def __init__(self, code: int, what: str = ""):
        self.code = code
        super().__init__(f"{what}: {ERRORS.get(code, code)} ({code})")


class GnnConfig(ctypes.Structure):
    _fields_ = [("version", ctypes.c_int32), ("n_node_feat", ctypes.c_int32),
                ("n_edge_feat", ctypes.c_int32), ("hidden", ctypes.c_int32),
                ("n_iters", ctypes.c_int32), ("mlp_layers", ctypes.c_int32),
                ("precision", ctypes.c_int32), ("ln_eps", ctypes.c_float)]


def load_library(path: str = LIB_PATH):
    """Load the CUDA library; raises when it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"CUDA library not built ({path}); run __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    lib.gnn_create.argtypes = [ctypes.POINTER(GnnConfig), vp, ctypes.c_size_t, ctypes.POINTER(vp)]
    lib.gnn_create.restype = i32
    lib.gnn_reserve.argtypes = [vp, i64, i64]
    lib.gnn_reserve.restype = i32
    lib.gnn_infer.argtypes = [vp, vp, vp, i64, i64, vp, vp]
    lib.gnn_infer.restype = i32
    lib.gnn_status.argtypes = [vp, vp]
    lib.gnn_status.restype = i32
    lib.gnn_destroy.argtypes = [vp]
    lib.gnn_destroy.restype = None
    lib.gnn_error_string.argtypes = [i32]
    lib.gnn_error_string.restype = ctypes.c_char_p
    lib.gnn_debug_copy.argtypes = [vp, i32, vp, ctypes.c_size_t, vp]
    lib.gnn_debug_copy.restype = i32
    lib.gnn_infer_host.argtypes = [vp, vp, vp, i64, i64, vp, vp]
    lib.gnn_infer_host.restype = i32
    lib.gnn_profile_enable.argtypes = [vp, i32]
    lib.gnn_profile_enable.restype = i32
    lib.gnn_profile_read.argtypes = [vp, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int64), i32]
    lib.gnn_profile_read.restype = i32
    lib.gnn_track_labels.argtypes = [vp, vp, vp, i64, i64, ctypes.c_float, vp, vp]
    lib.gnn_track_labels.restype = i32
    lib.gnn_filter_load.argtypes = [vp, vp, ctypes.c_size_t]
    lib.gnn_filter_load.restype = i32
    lib.gnn_filter_edges.argtypes = [vp, vp, vp, i64, i64, ctypes.c_float, vp, vp, vp, vp, vp]
    lib.gnn_filter_edges.restype = i32
    lib.gnn_embed_load.argtypes = [vp, vp, ctypes.c_size_t]
    lib.gnn_embed_load.restype = i32
    lib.gnn_embed.argtypes = [vp, vp, i64, vp, vp]
    lib.gnn_embed.restype = i32
    lib.gnn_build_graph.argtypes = [vp, vp, i32, vp, i64, ctypes.c_float, i64, vp, vp, vp]
    lib.gnn_build_graph.restype = i32
    _lib = lib
    return lib


def _stream_handle(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


class InteractionNetwork:
    """One library context: a model (config + weight blob) on the current device."""

    def __init__(self, model_cfg, blob: bytes):
        self.lib = load_library()
        self.cfg = model_cfg
        c = GnnConfig(1, model_cfg.n_node_feat, model_cfg.n_edge_feat, model_cfg.hidden,
                      model_cfg.n_iters, model_cfg.mlp_layers, model_cfg.precision, model_cfg.ln_eps)
        buf = ctypes.create_string_buffer(blob, len(blob))
        h = ctypes.c_void_p()
        rc = self.lib.gnn_create(ctypes.byref(c), buf, len(blob), ctypes.byref(h))
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_create")
        self.handle = h

    def reserve(self, n_nodes: int, n_edges: int):
        rc = self.lib.gnn_reserve(self.handle, n_nodes, n_edges)
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_reserve")

    def infer(self, x, edge_index, scores=None, stream=None):
        """x: cuda float32 [N, F_n]; edge_index: cuda int32 [2, E]; returns cuda float32 [E]."""
        import torch
        assert x.is_cuda and x.dtype == torch.float32 and x.is_contiguous()
        assert edge_index.is_cuda and edge_index.dtype == torch.int32 and edge_index.is_contiguous()
        E = edge_index.shape[1]
        if scores is None:
            scores = torch.empty(E, dtype=torch.float32, device=x.device)
        rc = self.lib.gnn_infer(self.handle, ctypes.c_void_p(x.data_ptr()),
                                ctypes.c_void_p(edge_index.data_ptr()), x.shape[0], E,
                                ctypes.c_void_p(scores.data_ptr()), _stream_handle(stream))
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_infer")
        return scores

    def infer_host(self, x, edge_index, scores, stream=None) -> int:
        """Host buffers in and out (numpy arrays or pinned CPU tensors); returns the status code."""
        import numpy as np

        def ptr(a):
            return ctypes.c_void_p(a.data_ptr() if hasattr(a, "data_ptr") else a.ctypes.data)
        n, e = x.shape[0], edge_index.shape[1]
        if isinstance(x, np.ndarray):
            assert x.dtype == np.float32 and edge_index.dtype == np.int32 and scores.dtype == np.float32
            assert x.flags.c_contiguous and edge_index.flags.c_contiguous
        rc = self.lib.gnn_infer_host(self.handle, ptr(x), ptr(edge_index), n, e, ptr(scores),
                                     _stream_handle(stream))
        if rc not in (GNN_OK, -5):
            raise GnnError(rc, "gnn_infer_host")
        return rc

    def track_labels(self, scores, edge_index, n_nodes: int, threshold: float = 0.5, labels=None,
                     stream=None):
        """Track candidates: int32 [n_nodes] cuda labels (smallest hit id of each connected
        component of the edges with score > threshold)."""
        import torch
        assert scores.is_cuda and scores.dtype == torch.float32 and scores.is_contiguous()
        assert edge_index.is_cuda and edge_index.dtype == torch.int32 and edge_index.is_contiguous()
        if labels is None:
            labels = torch.empty(n_nodes, dtype=torch.int32, device=scores.device)
        rc = self.lib.gnn_track_labels(self.handle, ctypes.c_void_p(scores.data_ptr()),
                                       ctypes.c_void_p(edge_index.data_ptr()), n_nodes, edge_index.shape[1],
                                       float(threshold), ctypes.c_void_p(labels.data_ptr()),
                                       _stream_handle(stream))
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_track_labels")
        return labels

    def load_embedding(self, blob: bytes):
        """Load the embedding MLP (blob of synthetic.pack_embed_blob)."""
        buf = ctypes.create_string_buffer(blob, len(blob))
        rc = self.lib.gnn_embed_load(self.handle, buf, len(blob))
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_embed_load")
        self.embed_dim = struct.unpack_from("<8i", blob)[6]

    def embed(self, x, stream=None):
        """Embedding [N, dim] (cuda float32) of every hit; dim is the loaded embedding MLP's."""
        import torch
        assert x.is_cuda and x.dtype == torch.float32 and x.is_contiguous()
        out = torch.empty((x.shape[0], getattr(self, "embed_dim", 1)), dtype=torch.float32, device=x.device)
        rc = self.lib.gnn_embed(self.handle, ctypes.c_void_p(x.data_ptr()), x.shape[0],
                                ctypes.c_void_p(out.data_ptr()), _stream_handle(stream))
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_embed")
        return out

    def build_graph(self, emb, x, radius: float, max_edges: int, stream=None):
        """Fixed-radius candidate edges: (edge index [2, n] cuda int32, n).  Raises GnnError
        (CAPACITY) when more than max_edges edges exist, with the number found as .n_edges."""
        import torch
        assert emb.is_cuda and emb.dtype == torch.float32 and emb.is_contiguous()
        out = torch.empty(2 * max(max_edges, 1), dtype=torch.int32, device=emb.device)
        n = torch.zeros(1, dtype=torch.int32, device=emb.device)
        rc = self.lib.gnn_build_graph(self.handle, ctypes.c_void_p(emb.data_ptr()), emb.shape[1],
                                      ctypes.c_void_p(x.data_ptr()), emb.shape[0], float(radius), max_edges,
                                      ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(n.data_ptr()),
                                      _stream_handle(stream))
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_build_graph")
        st = self.status(stream)
        k = int(n.item())
        if st != GNN_OK:
            err = GnnError(st, "gnn_build_graph")
            err.n_edges = k
            raise err
        return out[:2 * k].view(2, k), k

    def load_filter(self, blob: bytes):
        """Load the filtering MLP (blob of synthetic.pack_filter_blob)."""
        buf = ctypes.create_string_buffer(blob, len(blob))
        rc = self.lib.gnn_filter_load(self.handle, buf, len(blob))
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_filter_load")

    def filter_edges(self, x, edge_index, threshold: float = 0.5, stream=None):
        """Filtering step: (scores [E], kept edge index [2, n_kept], kept input ids [n_kept]),
        all cuda tensors; scores are the filter's, for every input edge."""
        import torch
        assert x.is_cuda and x.dtype == torch.float32 and x.is_contiguous()
        assert edge_index.is_cuda and edge_index.dtype == torch.int32 and edge_index.is_contiguous()
        E = edge_index.shape[1]
        scores = torch.empty(E, dtype=torch.float32, device=x.device)
        kept = torch.empty(2 * max(E, 1), dtype=torch.int32, device=x.device)
        kept_id = torch.empty(max(E, 1), dtype=torch.int32, device=x.device)
        n_kept = torch.zeros(1, dtype=torch.int32, device=x.device)
        rc = self.lib.gnn_filter_edges(self.handle, ctypes.c_void_p(x.data_ptr()),
                                       ctypes.c_void_p(edge_index.data_ptr()), x.shape[0], E, float(threshold),
                                       ctypes.c_void_p(scores.data_ptr()), ctypes.c_void_p(kept.data_ptr()),
                                       ctypes.c_void_p(kept_id.data_ptr()), ctypes.c_void_p(n_kept.data_ptr()),
                                       _stream_handle(stream))
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_filter_edges")
        n = int(n_kept.item())
        return scores, kept[:2 * n].view(2, n), kept_id[:n]

    def profile(self, on: bool = True):
        self.lib.gnn_profile_enable(self.handle, 1 if on else 0)

    def profile_read(self) -> dict:
        n = len(PROFILE_GROUPS)
        ms = (ctypes.c_double * n)()
        cnt = (ctypes.c_int64 * n)()
        rc = self.lib.gnn_profile_read(self.handle, ms, cnt, n)
        if rc < 0:
            raise GnnError(rc, "gnn_profile_read")
        return {g: (ms[i], cnt[i]) for i, g in enumerate(PROFILE_GROUPS)}

    def status(self, stream=None) -> int:
        return self.lib.gnn_status(self.handle, _stream_handle(stream))

    def debug_copy(self, which: int, shape, dtype, stream=None):
        import torch
        out = torch.empty(shape, dtype=dtype, device="cuda")
        rc = self.lib.gnn_debug_copy(self.handle, which, ctypes.c_void_p(out.data_ptr()),
                                     out.numel() * out.element_size(), _stream_handle(stream))
        if rc != GNN_OK:
            raise GnnError(rc, "gnn_debug_copy")
        return out

    def close(self):
        if getattr(self, "handle", None):
            self.lib.gnn_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
