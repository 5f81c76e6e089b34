"""CPU oracle for the E-step / M-step of Variational Speculative Decoding.

TEST INFRASTRUCTURE ONLY.  Plain C in fp64 (vsd_oracle.c) behind a ctypes
front end (oracle.py).  Only tests/, the smoke check and the benchmark's
CPU-baseline leg may import it; the CUDA library never does, and the two share
no code.  Parity pins for every oracle function live in tests/test_oracle_*.py.
"""
