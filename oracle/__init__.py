"""CPU oracle for the retrieve-and-verify step.

Test infrastructure only: imported by tests/, __graft_entry__.smoke() and the
CPU-baseline leg of bench.py.  The product package never imports it.
"""
