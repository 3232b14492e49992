"""Plain CPU oracle for the SFC GEMM -- test infrastructure only (see oracle.py)."""
