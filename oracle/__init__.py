"""fp64 CPU oracle of the xHC connection op -- TEST INFRASTRUCTURE ONLY.

Only tests/, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
anything under ``oracle/``.  The product path never does.
"""
