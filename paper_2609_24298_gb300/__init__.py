"""KV-COBRA hot path on GB300 (sm_103a): a C-ABI library (libcobra.so, include/cobra.h) with
CUDA kernels for per-token compression and rank-space decode attention over a packed KV
cache, plus a thin ctypes binding (`cobra`), seeded synthetic inputs (`synth`) and a
pipeline that assembles a compressed cache through the library (`pipeline`)."""
from . import cobra, synth  # noqa: F401

__all__ = ["cobra", "synth"]
