"""GB300-native verification step of speculative cascades (arXiv 2405.19261).

The compute path is the C-ABI library ``libspeccascade.so`` (hand-written
sm_103a CUDA kernels); ``paper_2405_19261_gb300.binding`` marshals torch
tensors into it.  The library is loaded on first use and a missing or stale
build raises at that point: there is no CPU fallback.

``paper_2405_19261_gb300.sharded`` runs the same step with the vocabulary split
across GPUs (a tensor-parallel LM head), through the same library.

``paper_2405_19261_gb300.workloads`` draws seeded synthetic inputs and does not
touch the library.
"""

__all__ = ["sc_verify", "sc_row_stats", "workspace_bytes", "verify", "row_stats"]


def __getattr__(name):
    if name in __all__:
        from . import binding
        return getattr(binding, name)
    raise AttributeError(name)
