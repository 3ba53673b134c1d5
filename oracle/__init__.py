"""fp64 CPU oracle of FadeMem (arxiv 2606.10671): Algorithm S1 and cache attention.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference leg of ``bench.py`` import this package.  It shares no
code with the CUDA library in ``paper_2606_10671_gb300`` and imports nothing
from it.  See ``fademem_oracle.c`` for what each function computes and the
passage of the paper it follows.
"""
from .oracle import OracleMemory, build_oracle, oracle_num_threads, OP_WEIGHTED, OP_AVERAGE, \
    OP_SELECT_NEAREST, OP_MAX_POOL

__all__ = ["OracleMemory", "build_oracle", "oracle_num_threads", "OP_WEIGHTED", "OP_AVERAGE",
           "OP_SELECT_NEAREST", "OP_MAX_POOL"]
