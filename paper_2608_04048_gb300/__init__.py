"""GB300 (sm_103a) Recurrent Residual Quantization: fused CUDA construction of
the 2/4/6/8-bit RRQ package and its prefix reconstruction, behind a C ABI
(include/rrq.h) with a thin ctypes binding.

Importing the package loads nothing; the CUDA library is loaded on the first
call of rrq_quantize / rrq_reconstruct and a missing library is an error.
"""
from .binding import (Package, RRQError, library_path, load_library, rrq_codes_bytes,
                      rrq_get_device_status, rrq_meta_count, rrq_package_bytes,
                      rrq_quantize, rrq_quantize_batch, rrq_reconstruct, rrq_reconstruct_batch,
                      rrq_reconstruct_prefixes, rrq_reconstruct_prefixes_batch,
                      rrq_set_debug_flags, rrq_set_wait_limit_us)

__all__ = ["Package", "RRQError", "library_path", "load_library", "rrq_codes_bytes",
           "rrq_get_device_status", "rrq_meta_count", "rrq_package_bytes", "rrq_quantize",
           "rrq_quantize_batch", "rrq_reconstruct", "rrq_reconstruct_batch", "rrq_reconstruct_prefixes",
           "rrq_reconstruct_prefixes_batch", "rrq_set_debug_flags",
           "rrq_set_wait_limit_us"]
