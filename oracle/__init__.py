"""CPU oracle for the selective-recompute prefill (test infrastructure only).

This package is the plain, slow, obviously-correct statement of what the CUDA
path computes.  It is test infrastructure: only `tests/`, the smoke check in
`__graft_entry__.py` and the `cpu_baseline` / reference leg of `bench.py` may
import it.  The product path never calls it and shares no code with it.

Arithmetic is float64 numpy throughout (inputs are bf16-representable values
upcast to float64).  Library primitives used as single steps: `numpy.matmul`
(for Linear layers and attention scores), `numpy.exp`, `numpy.argsort`.

Modules
  llama  - one Llama-3.1 decoder layer over an arbitrary set of rows attending a
           KV cache (RMSNorm, QKV, RoPE with llama3 frequency scaling, causal GQA
           attention, O-proj, SwiGLU MLP).
  blend  - the method (Sec. 3.2, Sec. 3.4, Sec. 4): per-chunk caches, RoPE
           re-alignment, HKVD deviation and top-k selection, selective prefill,
           and the full causal prefill it is compared against.

Parity status: every function here is pinned by `tests/test_oracle_*.py`
against closed forms, library routines, invariants the paper states and brute
force on tiny inputs; none is "parity unpinned".
"""
from . import llama, blend  # noqa: F401
