"""SFC GEMM for GB300: generalized-Hilbert-ordered, communication-avoiding bf16
GEMM on sm_103a tensor cores, exposed through a C ABI (``include/sfc_gemm.h``)
and this thin ctypes binding.  See ``binding.py`` for the Python entry points."""
from .binding import (SfcError, SfcLibraryMissing, debug_force_timeout, device_status, gemm, gemm_host, gemm_raw,
                      load, matmul_host, mma_peak, num_workers, plan, release, tile_order, tile_order_device,
                      tune, tune_forget, tune_lookup, workspace_size)

__all__ = ["SfcError", "SfcLibraryMissing", "debug_force_timeout", "device_status", "gemm", "gemm_host", "gemm_raw",
           "load", "matmul_host", "mma_peak", "num_workers", "plan", "release", "tile_order", "tile_order_device",
           "tune", "tune_forget", "tune_lookup", "workspace_size"]
