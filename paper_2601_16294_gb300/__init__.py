"""SFC GEMM for GB300 (placeholder; the CUDA binding is added with the library)."""
