"""Exact Minimum-Prefix-Trie solver for GB300 (sm_103a).

"Prefix Sharing Is a Sorting Problem" (arxiv 2609.13692) shows that the least
prefill cost of laying out request chunk sets for an exact-prefix KV cache is
a minimum over binary hierarchies on the requests (Thm 1), computed exactly
by an O(3^m) subset recurrence (Sec. 3.1).  This package runs that recurrence
in hand-written CUDA kernels behind the C ABI of ``include/mpt.h``:

* ``mpt``        -- the ctypes binding (``mpt.solve(weights, bits)``);
* ``instances``  -- seeded synthetic instances (RAG-shaped pools, L_n, ...);
* ``build``      -- compiles ``csrc/`` into ``_build/libmpt.so``.

The binding is imported on first use so that ``instances`` stays usable
without the compiled library.
"""

import importlib

from . import instances

__all__ = ["instances", "mpt", "build"]


def __getattr__(name):
    if name in ("mpt", "build"):
        return importlib.import_module(f".{name}", __name__)
    raise AttributeError(name)
