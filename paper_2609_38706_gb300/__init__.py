"""GB300-native provenance-bound KV-cache keys.

Key derivation, longest-prefix lookup and store against a GPU-resident table,
implemented as hand-written CUDA kernels for sm_103a behind the C-ABI library
``libpk.so`` (declared in ``include/pk.h``).  ``pk`` is the thin Python
binding; ``workloads`` draws the seeded synthetic inputs.
"""
__all__ = ["pk", "workloads"]
