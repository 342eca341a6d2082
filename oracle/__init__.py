"""CPU oracle of the batched FCFS / LJF / ISJL simulator.

TEST INFRASTRUCTURE: only ``tests/``, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may import anything here.  The product path (the
``paper_2608_02244_gb300`` package) never imports it.
"""
