"""GB300 (sm_103a) implementation of the AtSpeed verification call (arXiv 2410.05165).

The CUDA library ``_build/libatspeed.so`` (sources in ``csrc/``, C ABI in ``include/atspeed.h``)
does all the work; ``binding`` marshals torch tensors into its calls.
"""
from .binding import (E_ARG, E_CUDA, E_OOM, E_SHAPE, E_STATE, E_TIMEOUT, OK, AtSpeedError, Context, DecodeOpts,
                      EXPORTS, LIB_PATH, NORM_FULL, NORM_MASKED, PLAIN_SAMPLE, PLAIN_TOPK, RELAXED, SD_RELAXED,
                      SD_STRICT, STRICT, load, op_attention, op_gemm, op_gemm_noalloc, op_gemm_swiglu, op_rmsnorm,
                      op_status, opts, weights_to_device)

__all__ = ["E_ARG", "E_CUDA", "E_OOM", "E_SHAPE", "E_STATE", "E_TIMEOUT", "OK", "AtSpeedError", "Context", "DecodeOpts", "EXPORTS", "LIB_PATH", "NORM_FULL", "NORM_MASKED", "PLAIN_SAMPLE",
           "PLAIN_TOPK", "RELAXED", "SD_RELAXED", "SD_STRICT", "STRICT", "load", "op_attention", "op_gemm", "op_gemm_noalloc",
           "op_gemm_swiglu", "op_rmsnorm", "op_status", "opts", "weights_to_device"]
