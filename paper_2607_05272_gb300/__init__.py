"""GB300-native batched rollout engine for adaptive inference batching.

The compute path is the CUDA library ``libsimx.so`` (built from ``csrc/`` for
sm_103a); ``simx`` is its thin ctypes binding and ``workloads`` holds the seeded
synthetic inputs.  Importing the package does not load the library; the first call
into ``simx`` does, and fails loudly when it is missing.
"""
__all__ = ["simx", "workloads"]
