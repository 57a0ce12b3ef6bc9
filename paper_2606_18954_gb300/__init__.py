"""GB300-native GraphPO advantage construction.

Sampled rollout groups (step boundaries, state embeddings, binary rewards, step
lengths) -> per-token fp32 advantages, computed by the CUDA kernels of
libgraphpo (include/graphpo.h) on one sm_103a GPU.
"""
from .binding import (FLAG_SIMT_SIMILARITY, FLAG_TILED, Batch, GraphPO, GraphPOError,  # noqa: F401
                      load)
from .buildlib import build  # noqa: F401

__all__ = ["Batch", "GraphPO", "GraphPOError", "build", "load", "FLAG_SIMT_SIMILARITY", "FLAG_TILED"]
