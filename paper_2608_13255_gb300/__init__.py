"""GB300-native geometric delta transport (GeoCache, Sec. 3.2).

The compute path is the C-ABI library ``libgeocache.so`` (CUDA kernels for
sm_103a); :mod:`paper_2608_13255_gb300.geocache` is its ctypes binding and is
imported lazily so that the seeded input module
:mod:`paper_2608_13255_gb300.synth` can be used on machines without a GPU.
"""
__all__ = ["geocache", "synth"]


def __getattr__(name):
    if name in ("geocache", "synth"):
        import importlib
        return importlib.import_module(__name__ + "." + name)
    raise AttributeError(name)
