"""libunisvq: GB300 (sm_103a) kernels for the UniSVQ 2-bit linear layer.

The compute path is the C-ABI library `_lib/libunisvq.so` (include/unisvq.h);
`binding` wraps it with ctypes. Importing this package does not load the
library; `binding.load()` does, and raises if it has not been built.
"""
from .binding import (KERNEL_AUTO, KERNEL_DECODE, KERNEL_GEMV, KERNEL_PREFILL, KERNEL_SKINNY, UniSVQLinear, UnisvqError,  # noqa: F401
                      load, pack_host, packed_code_bytes, sync_status)

__all__ = ["UniSVQLinear", "UnisvqError", "load", "pack_host", "packed_code_bytes", "sync_status",
           "KERNEL_AUTO", "KERNEL_DECODE", "KERNEL_PREFILL", "KERNEL_GEMV", "KERNEL_SKINNY"]
