"""fp64 CPU oracle of the decode hot path -- test infrastructure only.

Used by tests/, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py``.  The product package never imports it.
"""
