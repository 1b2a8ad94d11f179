"""GB300 (sm_103a) implementation of the CRVQ code-search hot path (arXiv 2412.09282).

The compute runs in libcrvq.so (hand-written CUDA behind a C ABI, declared in include/crvq.h).
This package is a thin ctypes binding over it: functions keep the C names and only marshal
torch tensors (device memory and streams) into pointers and sizes. Nothing here computes a
step of the method on the host; if the library is missing, importing `api` raises.
"""
from .api import (  # noqa: F401
    Codebook, LayerOutputs, crvq_avg_bits, crvq_avg_bits_bases, crvq_coupled_sweep, crvq_encode_beam, crvq_hessian,
    crvq_hessian_blocks, crvq_hessian_inverse_diag,
    crvq_kmeans_init, crvq_lut_matvec, crvq_n_crit_groups, crvq_quantize_layer,
    crvq_reconstruct_error,
    crvq_select_reorder_channels, crvq_sync, crvq_update_codebook_noalloc, crvq_profile_begin,
    crvq_profile_end, crvq_profile_filter, crvq_launch_count, crvq_selftest_bounded_wait,
    crvq_update_codebook,
    crvq_version, CrvqError, IMPORTANCE_WA, IMPORTANCE_W_ONLY, IMPORTANCE_RANDOM,
    IMPORTANCE_WA_INV, library_path,
)
