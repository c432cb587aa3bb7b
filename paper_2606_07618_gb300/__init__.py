"""GB300-native NVFP4 ScaleSweep quantisation.

The compute path is the C-ABI library ``libnvfp4ss.so`` (hand-written CUDA for
sm_103a, declared in ``include/nvfp4ss.h``); ``binding`` marshals torch tensors
into its entry points.  ``workloads`` draws the seeded synthetic inputs.
Nothing here falls back to a CPU implementation: if the extension is missing,
the binding raises.
"""
import importlib

__all__ = ["binding", "workloads"]


def __getattr__(name):
    if name in __all__:
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
