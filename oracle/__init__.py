"""fp64 CPU oracle for the EC²MoE MoE-layer forward.

TEST INFRASTRUCTURE: imported only by tests/, ``__graft_entry__.smoke()`` and
the CPU-baseline / reference legs of ``bench.py``.  The product path (the
C-ABI library and its binding) never imports or calls it.
"""
