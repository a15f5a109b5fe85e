"""fp64 CPU oracle for the Sparse-Reslim routed encoder (arxiv 2607.02829).

TEST INFRASTRUCTURE ONLY.  The tests, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` are the only code allowed to
import it.  It shares no code with the CUDA library and imports nothing from
it.  See ``oracle/reslim.py`` for what each function computes and where the
paper defines it.
"""
from . import reslim  # noqa: F401
