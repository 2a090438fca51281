"""GB300 interaction-network edge classifier (edge classification of GNN-based tracking).

The compute path is the CUDA library ``libgnn_gb300.so`` built from ``csrc/``;
``binding`` wraps its C ABI (include/gnn.h) with ctypes.  There is no CPU
fallback: using the binding without the built library raises."""
from .binding import InteractionNetwork, GnnError, load_library  # noqa: F401
