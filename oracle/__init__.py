"""LayerCheck reference oracle -- TEST INFRASTRUCTURE ONLY.

A plain, slow CPU restatement of the paper's method (§3.2-§3.6) used to
check the CUDA path.  Only the tests, the smoke check and the benchmark's
CPU-baseline leg import it; the product package never does.
"""
