"""The oracle: test infrastructure only.

A plain, slow, single-threaded CPU reference of the rollout engine, written from
the paper ("Adaptive Inference Batching using Policy Gradients"): the event
simulator and policy in C (``oracle.c``, fp32 where the GPU takes the same integer
decisions in fp32) and the returns / GAE / loss gradients in numpy fp64
(``rl.py``).  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s
``cpu_baseline`` leg may import it.  It shares no code with the CUDA library.
"""
from .binding import (  # noqa: F401
    OracleEnv,
    build,
    detcos2pi,
    detexp,
    detlog,
    dettanh,
    duration,
    gridq,
    lib,
    make_config,
    map_fn,
    normal,
    obs_dim,
    philox,
    philox_n,
    policy,
    rollout,
    samplers,
    state_words,
)
