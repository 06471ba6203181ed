"""fp64 CPU oracle for the Nexus splice / re-rotate / suffix-attention path,
a plain model of the L0 exact-token radix arena, and one of the INT8 tool scan
with its margin gate.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline / reference arm of ``bench.py`` may import this package. It shares no
code with the CUDA library, and the product path never calls it.
"""
from .nexus_oracle import *  # noqa: F401,F403
from .nexus_oracle import __all__ as _core_all
from .warm_arena import *  # noqa: F401,F403
from .warm_arena import __all__ as _arena_all
from .slb import *  # noqa: F401,F403
from .slb import __all__ as _slb_all

__all__ = list(_core_all) + list(_arena_all) + list(_slb_all)
