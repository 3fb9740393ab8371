"""CPU oracle for the GSQ step.  TEST INFRASTRUCTURE ONLY.

Plain numpy restatement of the method (float64 arithmetic) used to check the
CUDA path.  Only tests, `__graft_entry__.smoke()` and the benchmark's
CPU-baseline leg may import this package; the product path never does.
"""
