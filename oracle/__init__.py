"""CPU oracle for the DQT BitLinear training step (test infrastructure only).

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The CUDA library and its Python binding
never import it.
"""
from .oracle import *  # noqa: F401,F403
