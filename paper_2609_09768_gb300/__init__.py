"""GB300-native selective-recompute prefill after KV-cache concatenation.

`kvblend`  - ctypes binding of libkvblend.so (the C ABI in include/kvblend.h)
`build`    - nvcc build of the library for sm_103a
`synth`    - seeded synthetic inputs (shapes, weights, tokens, chunk layout)
`workload` - device-side set-up of a request (weights, per-chunk caches) via the library

Submodules are imported on use so that `synth` can be loaded without the library.
"""
__all__ = ["kvblend", "build", "synth", "workload"]
