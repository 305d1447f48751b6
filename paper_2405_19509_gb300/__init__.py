"""GB300 gradient coding for partial stragglers: Python binding of libgc.so.

The functions here carry the C-ABI's names (include/gc.h) and only marshal
arguments: torch CUDA tensors become device pointers, the current torch
stream becomes the cudaStream_t, and workspaces are allocated with torch.
Every step of the computation runs in the CUDA kernels of libgc.so; if the
library is missing, importing this package raises.
"""
from .binding import (  # noqa: F401
    GC_BF16,
    GC_CYCLIC,
    GC_EXPLICIT,
    GC_F32,
    GC_LOGISTIC,
    GC_LSQ,
    GCError,
    Workspace,
    block_length,
    gc_chunk_grads,
    gc_chunk_grads_workspace,
    gc_coeff_workspace,
    gc_decode_batch,
    gc_decode_batch_workspace,
    gc_decode_apply,
    gc_decode_combine,
    gc_decode_plan,
    gc_decode_combine_workspace,
    gc_kernel_launches,
    gc_decode_tx,
    gc_encode,
    gc_encode_with_coeffs,
    gc_encode_workspace,
    gc_find_encoding_coeff,
    gc_last_error,
    gc_make_assignment,
    gc_mse,
    gc_mse_workspace,
    gc_set_wait_limit,
    gc_chunk_ordering,
    gc_trigger_times,
    gc_chunk_grads_batched,
    gc_decode_prepare,
    gc_decode_plan_prepared,
    gc_inject_stall,
    GC_STALL_CHUNK_GRADS,
    GC_STALL_COMBINE,
    GC_STALL_BATCHED,
    gc_sgd_step,
    gc_status,
    gc_version,
    lib,
    library_path,
)
