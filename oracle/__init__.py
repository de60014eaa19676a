"""CPU oracle for the HeRo routed FFN stack (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may import
anything under this package.  The CUDA product path never does.
"""
